// ff.cuh -- float-float ("double-single") accumulation for Eq. (1) without
// fp64 arithmetic.
//
// GB300 issues fp64 FMA/add at ~0.5 T instr/s and f32<->f64 / i64->f32
// conversions at ~0.6 T/s, against ~35 T/s for fp32 FMA.  The per-kernel work
// therefore stays in fp32 pairs: a value is hi + lo with |lo| <= ulp(hi)/2,
// about 48 significant bits.  Products use the FMA error term (Dekker's
// product), sums use Knuth's two-sum followed by Dekker's fast two-sum
// renormalisation.  Weights (durations) and weight sums stay exact in int64.
// The final doubles are assembled from the pair with integer operations only.
//
// Accuracy: each accumulation step adds a relative error of about 2^-47 of
// the running sum, so n terms stay within n * 2^-47 (1e-9 up to ~140k terms
// per operator; the long-op path splits sums into blocks).  Every helper
// assumes finite inputs; NaN and infinity are filtered before.
#pragma once
#include <stdint.h>

namespace opattr {

struct ff {
    float hi, lo;
};

// s + e == a + b exactly (Knuth two-sum, no magnitude precondition)
__device__ __forceinline__ ff two_sum(float a, float b) {
    float s = __fadd_rn(a, b);
    float bb = __fsub_rn(s, a);
    float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return ff{s, e};
}
// s + e == a + b exactly when |a| >= |b| (Dekker fast two-sum)
__device__ __forceinline__ ff fast_two_sum(float a, float b) {
    float s = __fadd_rn(a, b);
    float e = __fsub_rn(b, __fsub_rn(s, a));
    return ff{s, e};
}
// acc += (xh + xl)
__device__ __forceinline__ void ff_add(ff &acc, float xh, float xl) {
    ff s = two_sum(acc.hi, xh);
    float e = __fadd_rn(s.lo, __fadd_rn(acc.lo, xl));
    acc = fast_two_sum(s.hi, e);
}
// m * (dh + dl) as a pair (product error from the FMA, m*dl rounded once)
__device__ __forceinline__ ff ff_mul_f(float m, ff d) {
    float p = __fmul_rn(m, d.hi);
    float pe = __fmaf_rn(m, d.hi, -p);
    float pl = __fmaf_rn(m, d.lo, pe);
    return ff{p, pl};
}

// Non-negative int64 as a pair: exact below 2^48, else within 2^-48.
__device__ __forceinline__ ff ff_from_i64(long long d) {
    unsigned long long u = (unsigned long long)d;
    if (u < (1ull << 48)) {
        float a = __uint2float_rn((unsigned)(u >> 24)) * 16777216.0f;   // exact: < 2^24 times 2^24
        float b = __uint2float_rn((unsigned)(u & 0xFFFFFFu));            // exact: < 2^24
        return two_sum(a, b);
    }
    int s = 64 - __clzll(u) - 24;
    unsigned long long A = u >> s, B = u - (A << s);
    float a = ldexpf(__uint2float_rn((unsigned)A), s);
    float b = __ull2float_rn(B);
    return two_sum(a, b);
}

// A finite float as a signed integer significand m and exponent e: x = m * 2^e.
__device__ __forceinline__ int f32_decompose(float x, int *e) {
    unsigned u = __float_as_uint(x);
    int ex = (int)((u >> 23) & 0xFF);
    int m = (int)(u & 0x7FFFFF);
    if (ex == 0) *e = -149; else { m |= 0x800000; *e = ex - 150; }
    return (u >> 31) ? -m : m;
}

// Nearest double to acc * 2^F (round to nearest even), built from bits.
__device__ __forceinline__ double i64_scaled_to_f64(long long acc, int F) {
    if (acc == 0) return 0.0;
    unsigned long long sign = acc < 0 ? 1ull : 0ull;
    unsigned long long u = sign ? (unsigned long long)(-acc) : (unsigned long long)acc;
    int top = 63 - __clzll(u);
    int E = F + top;
    unsigned long long m;
    if (top > 52) {
        int s = top - 52;
        unsigned long long rem = u & ((1ull << s) - 1), half = 1ull << (s - 1);
        m = u >> s;
        if (rem > half || (rem == half && (m & 1ull))) {
            m++;
            if (m == (1ull << 53)) { m >>= 1; E++; }
        }
    } else {
        m = u << (52 - top);
    }
    unsigned long long bits = (sign << 63) | ((unsigned long long)(E + 1023) << 52) | (m & ((1ull << 52) - 1));
    return __longlong_as_double((long long)bits);
}

__device__ __forceinline__ double f32_to_f64_bits(float x) {
    int e;
    int m = f32_decompose(x, &e);
    return i64_scaled_to_f64((long long)m, e);
}

// hi + lo as the nearest double (within one ulp when |lo| <= ulp(hi)).
__device__ __forceinline__ double ff_to_f64(ff v) {
    int eh, el;
    int mh = f32_decompose(v.hi, &eh);
    int ml = f32_decompose(v.lo, &el);
    if (mh == 0) return f32_to_f64_bits(v.lo);
    const int F = eh - 38;
    long long acc = (long long)mh << 38;
    int sh = el - F;
    if (ml != 0) {
        if (sh >= 0 && sh <= 38) acc += (long long)ml << sh;
        else if (sh < 0 && sh > -63) acc += ((long long)ml) >> (-sh);
    }
    return i64_scaled_to_f64(acc, F);
}

// (n.hi + n.lo) / D for an int64 D > 0, as the nearest double (within a few
// units of 2^-46 relative).
__device__ __forceinline__ double ff_div_i64_to_f64(ff n, long long D) {
    ff d = ff_from_i64(D);
    float q1 = __fdiv_rn(n.hi, d.hi);
    float p = __fmul_rn(q1, d.hi);
    float pe = __fmaf_rn(q1, d.hi, -p);
    float p2 = __fmul_rn(q1, d.lo);
    float r = __fadd_rn(__fsub_rn(__fsub_rn(__fsub_rn(n.hi, p), pe), p2), n.lo);
    float q2 = __fdiv_rn(r, d.hi);
    return ff_to_f64(fast_two_sum(q1, q2));
}

}  // namespace opattr
