// tc_stage.cu -- one batch-shared 5-qubit stage on the tensor cores (tcgen05),
// measured against the same stage on the FP32 CUDA cores.
//
// A stage of K = 5 fused single-qubit runs whose matrices do not depend on the
// sample (shared weights) is the dense 32 x 32 complex matrix
// U = U_4 (x) U_3 (x) U_2 (x) U_1 (x) U_0 on the five low qubits; over a batch it
// is one matrix product: with the states cut into rows of 32 amplitudes
// (the other n - 5 qubits index the rows), psi'[row] = U psi[row].  This is the
// prior art's gate application by batched matrix multiplication (paper, Sec. 3
// "Gate Application and Differentiation": gates applied by reshaping the
// state and multiplying), here as a candidate for GB300's tensor cores.  In
// real form (interleaved re, im) it is D[rows x 64] = A[rows x 64] * W[64 x 64].
//
// Tensor-core form (tc_stage_kernel): each CTA owns tiles of 128 rows.  A and W
// are split into tf32 high and low parts (a = a_hi + a_lo, each exact in tf32's
// 10 explicit mantissa bits) and D = A_hi W_hi + A_hi W_lo + A_lo W_hi is
// accumulated in FP32 in tensor memory by tcgen05.mma kind::tf32 (M = 128,
// N = 64, K = 8 per instruction, 24 instructions per tile), issued by one
// thread; operands sit in shared memory in the canonical K-major layout without
// swizzle (8-row x 16-byte core matrices).  Each warp then reads its 32 rows
// back with tcgen05.ld and re-splits them for the next application.
//
// FP32 form (fp32_stage_kernel): each thread holds one row (32 amplitudes) in
// registers and applies the five 2x2 runs with packed FP32 (FFMA2), exactly as
// the sweep kernels apply a K = 5 register block.
//
// Both kernels apply the stage `repeats` times to data that stays on chip
// between applications, so the comparison measures arithmetic, not HBM.
// Every wait on the tensor cores is bounded: on timeout the kernel records an
// error and still releases its tensor memory.
#include <cuda_runtime.h>

#include <string>

#include "engine.h"
#include "sweep.cuh"

namespace vqc {
vqc_status set_error(vqc_status s, const std::string& msg);
}

namespace {

using namespace vqc;

constexpr int kRows = 128;            // rows per tile (MMA M)
constexpr int kCols = 64;             // reals per row (32 complex)
constexpr int kTmemCols = 256;        // allocated tensor-memory columns (>= N = 64)
constexpr unsigned kSpinLimit = 1u << 24;   // polls (about a second)

struct StageArgs {
    float f[5][8];          // the five 2x2 factors, row-major (re, im); factor q acts on qubit q
    const float2* in;
    float2* out;
    long long rows;         // batch * 2^(n - 5)
    int repeats;
    unsigned* err;          // error word: 1 = tensor-core wait timed out
};

// Byte offset of element (r, k) of a K-major operand in the no-swizzle
// canonical layout: 8-row x 4-element core matrices of 128 bytes, core (g, c)
// at (g * 16 + c) * 128 for 16 K-chunks of 4 tf32 values per row group.
__device__ __forceinline__ uint32_t core_off(int r, int k) {
    return (uint32_t)((((r >> 3) * 16 + (k >> 2)) << 7) + ((r & 7) << 4) + ((k & 3) << 2));
}

// tf32 rounding of an FP32 value (round to nearest, ties away; the MMA ignores
// the 13 low mantissa bits)
__device__ __forceinline__ float to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
    return __uint_as_float(r);
}

// Shared-memory matrix descriptor (tcgen05): start address, leading-dimension
// byte offset (next core matrix along K), stride byte offset (next 8-row
// group), descriptor version 1, no swizzle.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFF) >> 4) | ((uint64_t)((lbo & 0x3FFFF) >> 4) << 16) |
           ((uint64_t)((sbo & 0x3FFFF) >> 4) << 32) | ((uint64_t)1 << 46);
}

// Instruction descriptor, kind::tf32: FP32 accumulator, A and B tf32, both
// K-major, N = 64, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(kCols >> 3) << 17) |
                            ((uint32_t)(kRows >> 4) << 24);

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mma_tf32(uint32_t tmem, uint64_t a, uint64_t b, int accumulate) {
    asm volatile(
        "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem),
        "l"(a), "l"(b), "r"(kIdesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t mbar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(mbar)
                 : "memory");
}

// Wait for the mbarrier phase with the given parity; false after kSpinLimit polls.
__device__ __forceinline__ bool mbar_wait(uint32_t mbar, uint32_t parity) {
    for (unsigned it = 0; it < kSpinLimit; ++it) {
        uint32_t done;
        asm volatile(
            "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
            "selp.b32 %0, 1, 0, p;\n}\n"
            : "=r"(done)
            : "r"(mbar), "r"(parity)
            : "memory");
        if (done) return true;
    }
    return false;
}

// 16 consecutive FP32 accumulator columns of this warp's 32 lanes.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
        "%12, %13, %14, %15}, [%16];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}

constexpr int kSmemW = 16384, kSmemA = 32768;
constexpr int kSmemBytes = 2 * kSmemW + 2 * kSmemA + 64;

__global__ void __launch_bounds__(128, 1) tc_stage_kernel(const __grid_constant__ StageArgs A) {
    extern __shared__ __align__(1024) unsigned char sm[];
    unsigned char* wh = sm;
    unsigned char* wl = sm + kSmemW;
    unsigned char* ah = sm + 2 * kSmemW;
    unsigned char* al = sm + 2 * kSmemW + kSmemA;
    uint64_t* mbar = reinterpret_cast<uint64_t*>(sm + 2 * kSmemW + 2 * kSmemA);
    uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + 2 * kSmemW + 2 * kSmemA + 16);
    const int tid = threadIdx.x, warp = tid >> 5;

    // B operand: W^T[n][k] (n output real, k input real) of the dense 32 x 32
    // complex U, split into tf32 high and low parts, K-major core layout
    for (int idx = tid; idx < kCols * kCols; idx += blockDim.x) {
        const int n = idx / kCols, k = idx % kCols, ko = n >> 1, ki = k >> 1;
        float ur = 1.f, ui = 0.f;
#pragma unroll
        for (int q = 0; q < 5; ++q) {
            const int e = (((ko >> q) & 1) * 2 + ((ki >> q) & 1)) * 2;
            const float mr = A.f[q][e], mi = A.f[q][e + 1];
            const float tr = ur * mr - ui * mi, ti = ur * mi + ui * mr;
            ur = tr;
            ui = ti;
        }
        const float v = (n & 1) == 0 ? ((k & 1) == 0 ? ur : -ui) : ((k & 1) == 0 ? ui : ur);
        const float hi = to_tf32(v);
        *reinterpret_cast<float*>(wh + core_off(n, k)) = hi;
        *reinterpret_cast<float*>(wl + core_off(n, k)) = to_tf32(v - hi);
    }
    const uint32_t mb = smem_u32(mbar);
    if (tid == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(mb) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(tslot)),
                     "n"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t a_hi = smem_u32(ah), a_lo = smem_u32(al), w_hi = smem_u32(wh), w_lo = smem_u32(wl);
    uint32_t parity = 0;
    int ok = 1;
    for (long long t0 = (long long)blockIdx.x * kRows; t0 < A.rows && ok; t0 += (long long)gridDim.x * kRows) {
        const long long row = t0 + tid;
        float v[kCols];
        if (row < A.rows) {
            const float4* src = reinterpret_cast<const float4*>(A.in + row * 32);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const float4 x = src[i];
                v[4 * i] = x.x; v[4 * i + 1] = x.y; v[4 * i + 2] = x.z; v[4 * i + 3] = x.w;
            }
        } else {
#pragma unroll
            for (int i = 0; i < kCols; ++i) v[i] = 0.f;
        }
        for (int rep = 0; rep < A.repeats; ++rep) {
#pragma unroll
            for (int k = 0; k < kCols; k += 4) {   // this thread's row, high and low parts
                float4 h, l;
                h.x = to_tf32(v[k]); h.y = to_tf32(v[k + 1]); h.z = to_tf32(v[k + 2]); h.w = to_tf32(v[k + 3]);
                l.x = to_tf32(v[k] - h.x); l.y = to_tf32(v[k + 1] - h.y);
                l.z = to_tf32(v[k + 2] - h.z); l.w = to_tf32(v[k + 3] - h.w);
                *reinterpret_cast<float4*>(ah + core_off(tid, k)) = h;
                *reinterpret_cast<float4*>(al + core_off(tid, k)) = l;
            }
            asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
            tc_fence_before();
            __syncthreads();
            tc_fence_after();
            if (tid == 0) {
                // K = 8 per instruction: k-step s covers core chunks 2s, 2s + 1
                for (int s = 0; s < kCols / 8; ++s)
                    mma_tf32(tmem, smem_desc(a_hi + 256 * s, 128, 2048), smem_desc(w_hi + 256 * s, 128, 2048), s > 0);
                for (int s = 0; s < kCols / 8; ++s)
                    mma_tf32(tmem, smem_desc(a_hi + 256 * s, 128, 2048), smem_desc(w_lo + 256 * s, 128, 2048), 1);
                for (int s = 0; s < kCols / 8; ++s)
                    mma_tf32(tmem, smem_desc(a_lo + 256 * s, 128, 2048), smem_desc(w_hi + 256 * s, 128, 2048), 1);
                mma_commit(mb);
            }
            ok = __syncthreads_and(mbar_wait(mb, parity) ? 1 : 0);
            parity ^= 1;
            tc_fence_after();
            if (!ok) break;
            const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll
            for (int c = 0; c < kCols; c += 16) tmem_ld16(taddr + c, v + c);
            asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
            tc_fence_before();
            __syncthreads();   // every lane read before the next products overwrite D
        }
        if (ok && row < A.rows) {
            float4* dst = reinterpret_cast<float4*>(A.out + row * 32);
#pragma unroll
            for (int i = 0; i < 16; ++i) dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        }
    }
    if (!ok) {
        if (tid == 0) atomicOr(A.err, 1u);
        mbar_wait(mb, parity ^ 1);   // let products still in flight finish (bounded) before freeing
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "n"(kTmemCols)
                     : "memory");
}

// The same stage on the FP32 units: one row (32 amplitudes) per thread in
// registers, five packed-FP32 2x2 runs per application.
__global__ void __launch_bounds__(256, 2) fp32_stage_kernel(const __grid_constant__ StageArgs A) {
    __shared__ __align__(16) float tab[5][16];
    if (threadIdx.x < 5) {
        M2<float> m;
        const float* f = A.f[threadIdx.x];
        m.a = make_float2(f[0], f[1]); m.b = make_float2(f[2], f[3]);
        m.c = make_float2(f[4], f[5]); m.d = make_float2(f[6], f[7]);
        float t32[32];
        store_matrix<float>(m, t32);
        for (int i = 0; i < 16; ++i) tab[threadIdx.x][i] = t32[i];
    }
    __syncthreads();
    for (long long row = blockIdx.x * (long long)blockDim.x + threadIdx.x; row < A.rows;
         row += (long long)gridDim.x * blockDim.x) {
        float2 a[32];
        const float4* src = reinterpret_cast<const float4*>(A.in + row * 32);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float4 x = src[i];
            a[2 * i] = make_float2(x.x, x.y);
            a[2 * i + 1] = make_float2(x.z, x.w);
        }
        for (int rep = 0; rep < A.repeats; ++rep) {
            m1_apply_f2w<5, 0>(a, tab[0]);
            m1_apply_f2w<5, 1>(a, tab[1]);
            m1_apply_f2w<5, 2>(a, tab[2]);
            m1_apply_f2w<5, 3>(a, tab[3]);
            m1_apply_f2w<5, 4>(a, tab[4]);
        }
        float4* dst = reinterpret_cast<float4*>(A.out + row * 32);
#pragma unroll
        for (int i = 0; i < 16; ++i) dst[i] = make_float4(a[2 * i].x, a[2 * i].y, a[2 * i + 1].x, a[2 * i + 1].y);
    }
}

__device__ unsigned g_stage_err;

}  // namespace

namespace vqc {

// vqc_sync_check's view of the stage kernels' error word (read and cleared).
vqc_status stage_error_check() {
    unsigned e = 0;
    cudaError_t c = cudaMemcpyFromSymbol(&e, g_stage_err, sizeof(e));
    if (c != cudaSuccess) return set_error(VQC_ERR_CUDA, std::string("stage error word: ") + cudaGetErrorString(c));
    if (!e) return VQC_OK;
    const unsigned zero = 0;
    cudaMemcpyToSymbol(g_stage_err, &zero, sizeof(zero));
    return set_error(VQC_ERR_DEVICE_CHECK, "vqc_stage_apply: a tensor-core completion wait timed out");
}

}  // namespace vqc

extern "C" vqc_status vqc_stage_apply(int32_t method, int32_t batch, int32_t num_qubits, const double* factors,
                                      const void* psi_in, void* psi_out, int32_t repeats, void* stream) {
    try {
        if ((method != 0 && method != 1) || batch < 0 || num_qubits < 5 || num_qubits > VQC_MAX_QUBITS ||
            repeats < 1 || !factors || (batch > 0 && (!psi_in || !psi_out)))
            return set_error(VQC_ERR_INVALID_ARG, "vqc_stage_apply: bad method, batch, qubit count, "
                                                  "repeats or NULL pointer");
        if ((reinterpret_cast<uintptr_t>(psi_in) | reinterpret_cast<uintptr_t>(psi_out)) & 15)
            return set_error(VQC_ERR_INVALID_ARG, "vqc_stage_apply: state arrays must be 16-byte aligned");
        if (batch == 0) return VQC_OK;
        StageArgs a{};
        for (int q = 0; q < 5; ++q)
            for (int i = 0; i < 8; ++i) a.f[q][i] = (float)factors[8 * q + i];
        a.in = static_cast<const float2*>(psi_in);
        a.out = static_cast<float2*>(psi_out);
        a.rows = (long long)batch << (num_qubits - 5);
        a.repeats = repeats;
        void* ep = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&ep, g_stage_err);
        if (e != cudaSuccess) return set_error(VQC_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
        a.err = static_cast<unsigned*>(ep);
        int dev = 0, sms = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        cudaStream_t s = static_cast<cudaStream_t>(stream);
        void* args[] = {&a};
        if (method == 1) {
            e = cudaFuncSetAttribute((const void*)tc_stage_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     kSmemBytes);
            if (e != cudaSuccess) return set_error(VQC_ERR_CUDA, std::string("cudaFuncSetAttribute: ") + cudaGetErrorString(e));
            const long long tiles = (a.rows + kRows - 1) / kRows;
            const int grid = (int)std::min<long long>(tiles, sms);
            e = cudaLaunchKernel((const void*)tc_stage_kernel, dim3(grid), dim3(kRows), args, kSmemBytes, s);
        } else {
            const long long blocks = (a.rows + 255) / 256;
            const int grid = (int)std::min<long long>(blocks, (long long)sms * 8);
            e = cudaLaunchKernel((const void*)fp32_stage_kernel, dim3(grid), dim3(256), args, 0, s);
        }
        if (e != cudaSuccess) return set_error(VQC_ERR_CUDA, std::string("vqc_stage_apply launch: ") + cudaGetErrorString(e));
        return VQC_OK;
    } catch (...) {
        return set_error(VQC_ERR_INVALID_ARG, "internal error in vqc_stage_apply");
    }
}
