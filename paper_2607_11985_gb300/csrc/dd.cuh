// dd.cuh -- double-float ("float-float") arithmetic for the complex128 sweeps on
// the FP32 units.
//
// A value is the unevaluated sum hi + lo of two floats with |lo| <= ulp(hi)/2,
// about 48 significant bits.  The operations are the classical error-free
// transformations: Knuth's TwoSum (the exact rounding error of a sum, six
// additions, no ordering assumption), Dekker's FastTwoSum (three additions when
// |a| >= |b|) and the FMA form of the exact product (the rounding error of
// a*b is fma(a, b, -round(a*b))), combined as in Dekker's 1971 double-length
// arithmetic.  Every step is written with the _rn intrinsics, which the
// compiler never contracts into an FMA or reorders, so each transformation
// stays exact.  Relative error per operation is below 2^-44 (for sums whose
// terms cancel, the error is that fraction of the terms' magnitudes); with
// |amplitudes| <= 1 that is far below the 1e-10 absolute parity bound of the
// complex128 path.  The exponent range is float's: values below ~1e-30 lose
// low-part bits to subnormals (absolute error < 1e-38, irrelevant here).
//
// Storage stays complex128 (double, double2) everywhere outside the kernels:
// values are split when read (hi = double rounded to float, lo = the exact
// remainder rounded) and rejoined when written (hi + lo, exact in double).
#pragma once

#include <cuda_runtime.h>

namespace vqc {

struct __align__(8) dd {
    float hi, lo;
    dd() = default;
    __host__ __device__ constexpr dd(float h, float l) : hi(h), lo(l) {}
    __host__ __device__ constexpr dd(int v) : hi((float)v), lo(0.f) {}
    __host__ __device__ constexpr dd(float v) : hi(v), lo(0.f) {}
    __host__ __device__ explicit dd(double v) : hi((float)v), lo((float)(v - (double)(float)v)) {}

    __device__ __forceinline__ double to_double() const { return (double)hi + (double)lo; }

    friend __device__ __forceinline__ dd operator-(dd a) { return dd(-a.hi, -a.lo); }

    // hi + lo of a sum, TwoSum on the high parts, low parts added to the error
    friend __device__ __forceinline__ dd operator+(dd a, dd b) {
        const float s = __fadd_rn(a.hi, b.hi);
        const float v = __fsub_rn(s, a.hi);
        float e = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(s, v)), __fsub_rn(b.hi, v));
        e = __fadd_rn(e, __fadd_rn(a.lo, b.lo));
        const float h = __fadd_rn(s, e);
        return dd(h, __fsub_rn(e, __fsub_rn(h, s)));
    }
    friend __device__ __forceinline__ dd operator-(dd a, dd b) { return a + (-b); }

    // exact product of the high parts plus the cross terms
    friend __device__ __forceinline__ dd operator*(dd a, dd b) {
        const float p = __fmul_rn(a.hi, b.hi);
        float e = __fmaf_rn(a.hi, b.hi, -p);
        e = __fmaf_rn(a.hi, b.lo, e);
        e = __fmaf_rn(a.lo, b.hi, e);
        const float h = __fadd_rn(p, e);
        return dd(h, __fsub_rn(e, __fsub_rn(h, p)));
    }

    // a * b + c with one normalisation: the product's error terms join the
    // sum's TwoSum error before the final FastTwoSum
    friend __device__ __forceinline__ dd fma(dd a, dd b, dd c) {
        const float p = __fmul_rn(a.hi, b.hi);
        float pe = __fmaf_rn(a.hi, b.hi, -p);
        pe = __fmaf_rn(a.hi, b.lo, pe);
        pe = __fmaf_rn(a.lo, b.hi, pe);
        const float s = __fadd_rn(p, c.hi);
        const float v = __fsub_rn(s, p);
        float e = __fadd_rn(__fsub_rn(p, __fsub_rn(s, v)), __fsub_rn(c.hi, v));
        e = __fadd_rn(e, __fadd_rn(pe, c.lo));
        const float h = __fadd_rn(s, e);
        return dd(h, __fsub_rn(e, __fsub_rn(h, s)));
    }

    friend __device__ __forceinline__ dd& operator+=(dd& a, dd b) { return a = a + b; }
    friend __device__ __forceinline__ dd& operator-=(dd& a, dd b) { return a = a - b; }
    friend __device__ __forceinline__ dd& operator*=(dd& a, dd b) { return a = a * b; }
};

struct __align__(16) dd2 {
    dd x, y;
};

// a0 b0 + a1 b1 + a2 b2 + a3 b3 with a single normalisation (the compensated
// dot product of Ogita, Rump and Oishi, 2005): the high products are summed by
// TwoSum, every rounding error (of the sums, of the products, the cross terms
// hi*lo) is gathered in one float, and one FastTwoSum ends it.  43 FP32
// operations instead of 52 for a product and three fused multiply-adds.
__device__ __forceinline__ dd dot4(dd a0, dd b0, dd a1, dd b1, dd a2, dd b2, dd a3, dd b3) {
    float s = __fmul_rn(a0.hi, b0.hi);
    float err = __fmaf_rn(a0.hi, b0.hi, -s);
    err = __fmaf_rn(a0.hi, b0.lo, err);
    err = __fmaf_rn(a0.lo, b0.hi, err);
    const dd A[3] = {a1, a2, a3}, Bv[3] = {b1, b2, b3};
#pragma unroll
    for (int k = 0; k < 3; ++k) {
        const float p = __fmul_rn(A[k].hi, Bv[k].hi);
        const float e = __fmaf_rn(A[k].hi, Bv[k].hi, -p);
        const float t = __fadd_rn(s, p);
        const float v = __fsub_rn(t, s);
        const float r = __fadd_rn(__fsub_rn(s, __fsub_rn(t, v)), __fsub_rn(p, v));
        s = t;
        err = __fadd_rn(err, r);
        err = __fmaf_rn(A[k].hi, Bv[k].lo, err);
        err = __fmaf_rn(A[k].lo, Bv[k].hi, err);
        err = __fadd_rn(err, e);
    }
    const float h = __fadd_rn(s, err);
    return dd(h, __fsub_rn(err, __fsub_rn(h, s)));
}

}  // namespace vqc
