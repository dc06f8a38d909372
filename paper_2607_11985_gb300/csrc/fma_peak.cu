// fma_peak.cu -- vqc_fma_peak: the arithmetic ceiling of the sweep kernels,
// measured.
//
// The resident sweeps and the HBM passes spend their time in fused
// multiply-adds on the CUDA cores: packed FP32 pairs for complex64 states,
// FP64 for complex128.  Their roofline is the rate at which the device retires
// those instructions.  For FP32 it follows from the unit counts (128 lanes per
// SM, two flops per FMA); for FP64 the unit count of this part is not stated
// in any document at hand, so both are measured here with kernels that do
// nothing else: each thread runs eight independent FMA chains (enough
// independent work to cover the pipeline latency at full occupancy), the grid
// fills every SM, and the chains end in a comparison that the compiler cannot
// resolve, so no work is removed and nothing is written to memory.
#include <cuda_runtime.h>

#include <algorithm>
#include <string>

#include "vqc.h"

namespace vqc {
vqc_status set_error(vqc_status s, const std::string& msg);
}  // namespace vqc

namespace {

constexpr int kChains = 8;
constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads) fma_f32x2_kernel(int iters, float2 b, float2 c, float* sink) {
    float2 a[kChains];
#pragma unroll
    for (int i = 0; i < kChains; ++i)
        a[i] = make_float2(1e-3f * (float)threadIdx.x + (float)i, 1e-3f * (float)blockIdx.x - (float)i);
#pragma unroll 4
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int i = 0; i < kChains; ++i) a[i] = __ffma2_rn(a[i], b, c);
    }
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < kChains; ++i) s += a[i].x + a[i].y;
    if (s == -1.2345e-30f) sink[0] = s;
}

__global__ void __launch_bounds__(kThreads) fma_f64_kernel(int iters, double b, double c, double* sink) {
    double a[kChains];
#pragma unroll
    for (int i = 0; i < kChains; ++i) a[i] = 1e-3 * (double)threadIdx.x + (double)i - 1e-3 * (double)blockIdx.x;
#pragma unroll 4
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int i = 0; i < kChains; ++i) a[i] = fma(a[i], b, c);
    }
    double s = 0.0;
#pragma unroll
    for (int i = 0; i < kChains; ++i) s += a[i];
    if (s == -1.2345e-300) sink[0] = s;
}

}  // namespace

extern "C" vqc_status vqc_fma_peak(vqc_dtype dtype, double* tflops_out) {
    using vqc::set_error;
    if (!tflops_out) return set_error(VQC_ERR_INVALID_ARG, "tflops_out is NULL");
    if (dtype != VQC_C64 && dtype != VQC_C128 && dtype != VQC_C128_DF)
        return set_error(VQC_ERR_INVALID_ARG, "bad dtype");
    if (dtype == VQC_C128_DF) dtype = VQC_C64;   // double-float runs on the FP32 units
    *tflops_out = 0.0;
    int dev = 0, sms = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev);
    if (e != cudaSuccess) return set_error(VQC_ERR_CUDA, cudaGetErrorString(e));
    const bool dbl = dtype == VQC_C128;
    const int blocks = sms * std::max(1, per_sm / kThreads);
    // flops of one loop iteration over the whole grid: FMA = 2 flops, x2 lanes for the packed pair
    const double flops_per_iter = (double)blocks * kThreads * kChains * (dbl ? 2.0 : 4.0);
    void* sink = nullptr;
    cudaStream_t s = nullptr;
    cudaEvent_t t0 = nullptr, t1 = nullptr;
    double best = 0.0;
    auto run = [&](int iters, float* ms) -> cudaError_t {
        cudaError_t r = cudaEventRecord(t0, s);
        if (r != cudaSuccess) return r;
        if (dbl)
            fma_f64_kernel<<<blocks, kThreads, 0, s>>>(iters, 0.999999, 1e-7, static_cast<double*>(sink));
        else
            fma_f32x2_kernel<<<blocks, kThreads, 0, s>>>(iters, make_float2(0.9999f, 0.9999f),
                                                         make_float2(1e-4f, 1e-4f), static_cast<float*>(sink));
        if ((r = cudaGetLastError()) != cudaSuccess) return r;
        if ((r = cudaEventRecord(t1, s)) != cudaSuccess) return r;
        if ((r = cudaEventSynchronize(t1)) != cudaSuccess) return r;
        return cudaEventElapsedTime(ms, t0, t1);
    };
    e = cudaMalloc(&sink, 16);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreate(&t0);
    if (e == cudaSuccess) e = cudaEventCreate(&t1);
    if (e == cudaSuccess) {
        // calibrate on a short launch, then time launches of about 5 ms
        int iters = 256;
        float ms = 0.f;
        e = run(iters, &ms);
        if (e == cudaSuccess) {
            const double scale = 5.0 / std::max((double)ms, 1e-3);
            iters = (int)std::min(1.0e7, std::max(256.0, iters * scale));
            iters = (iters + 3) & ~3;
            for (int rep = 0; rep < 6 && e == cudaSuccess; ++rep) {
                e = run(iters, &ms);
                if (e == cudaSuccess && rep > 0 && ms > 0.f)
                    best = std::max(best, flops_per_iter * iters / (ms * 1e-3) / 1e12);
            }
        }
    }
    if (t1) cudaEventDestroy(t1);
    if (t0) cudaEventDestroy(t0);
    if (s) cudaStreamDestroy(s);
    if (sink) cudaFree(sink);
    if (e != cudaSuccess) return set_error(VQC_ERR_CUDA, cudaGetErrorString(e));
    *tflops_out = best;
    return VQC_OK;
}
