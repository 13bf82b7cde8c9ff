// ff.cuh -- float-float ("double-single") accumulation for Eq. (1) without
// fp64 arithmetic.
//
// GB300 issues fp64 FMA/add at ~0.5 T instr/s and f32<->f64 / i64->f32
// conversions at ~0.6 T/s, against ~35 T/s for fp32 FMA.  The per-kernel work
// therefore stays in fp32 pairs: a value is hi + lo, about 48 significant
// bits.  Products use the FMA error term (Dekker's product); sums use Knuth's
// two-sum into a running (hi, lo) pair whose lo collects the rounding errors
// and is folded back into hi (Dekker's fast two-sum) every RENORM terms and
// at the end.  Weights (durations) and weight sums stay exact in int64.  The
// final doubles are assembled from the pair with integer operations only.
//
// Accuracy: a step adds a relative error of about 2^-47 of the running sum,
// so n terms stay within n * 2^-47 (1e-9 for up to ~1.4e5 terms per
// operator).  Helpers assume finite inputs; NaN and infinity are filtered
// before.
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
// s + e == a + b exactly when |a| >= |b| or a == 0 (Dekker fast two-sum)
__device__ __forceinline__ ff fast_two_sum(float a, float b) {
    float s = __fadd_rn(a, b);
    float e = __fsub_rn(b, __fsub_rn(s, a));
    return ff{s, e};
}
// acc.hi + acc.lo += xh + xl, leaving lo unnormalised (see renorm)
__device__ __forceinline__ void ff_accum(ff &acc, float xh, float xl) {
    ff s = two_sum(acc.hi, xh);
    acc.hi = s.hi;
    acc.lo = __fadd_rn(acc.lo, __fadd_rn(s.lo, xl));
}
__device__ __forceinline__ void ff_renorm(ff &acc) {
    // |acc.lo| stays far below |acc.hi| between renormalisations unless the
    // running sum cancelled; two_sum keeps the pair exact either way
    acc = two_sum(acc.hi, acc.lo);
}

// Non-negative int64 as a normalised pair hi + lo (|lo| <= ulp(hi) / 2):
// exact below 2^48, within 2^-48 relative above.
__device__ __forceinline__ ff split_i64(long long d) {
    unsigned long long u = (unsigned long long)d;
    if (u < (1ull << 24)) return ff{__uint2float_rn((unsigned)u), 0.f};
    if (u < (1ull << 48)) {
        float a = __uint2float_rn((unsigned)(u >> 24)) * 16777216.0f;   // exact: the high 24 bits
        float b = __uint2float_rn((unsigned)(u & 0xFFFFFFu));            // exact: the low 24 bits
        return two_sum(a, b);
    }
    int s = 64 - __clzll(u) - 24;
    unsigned long long A = u >> s, B = u - (A << s);
    return two_sum(ldexpf(__uint2float_rn((unsigned)A), s), __ull2float_rn(B));
}

// m * (d.hi + d.lo) for a normalised d, as a pair: the first product exact
// through its FMA error, the second (2^-24 smaller) rounded once
__device__ __forceinline__ ff mul_split(float m, ff d) {
    float p = __fmul_rn(m, d.hi);
    float pe = __fmaf_rn(m, d.hi, -p);
    float pl = __fmaf_rn(m, d.lo, pe);
    return ff{p, pl};
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

// hi + lo as a double for a normalised pair (|lo| <= ulp(hi) / 2): hi's 24
// significand bits followed by lo's bits, truncated below 2^-53 of hi
// (within one double ulp).
__device__ __forceinline__ double ff_to_f64(ff v) {
    const unsigned uh = __float_as_uint(v.hi);
    const int exh = (int)((uh >> 23) & 0xFF);
    if (exh == 0) return f32_to_f64_bits(v.hi);       // zero or subnormal hi: a normalised lo is negligible
    int el;
    int ml = f32_decompose(v.lo, &el);
    if (uh >> 31) ml = -ml;                            // work on |hi|; lo enters with the relative sign
    // value = (mh * 2^29 + ml * 2^(el - (exh - 150) + 29)) * 2^(exh - 150 - 29)
    long long m = (long long)((uh & 0x7FFFFFu) | 0x800000u) << 29;
    const int sh = el - (exh - 150) + 29;
    if (ml != 0 && sh > -40) m += sh >= 0 ? ((long long)ml << sh) : ((long long)ml >> (-sh));
    // m is within a factor 2 of 2^52; renormalise by at most one bit
    int E = exh - 150 - 29 + 52;       // exponent of bit 52
    if (m >= (1ll << 53)) { m >>= 1; E++; }
    else if (m < (1ll << 52)) { m <<= 1; E--; }
    const unsigned long long bits = ((unsigned long long)(uh >> 31) << 63) | ((unsigned long long)(E + 1023) << 52) |
                                    ((unsigned long long)m & ((1ull << 52) - 1));
    return __longlong_as_double((long long)bits);
}

// The rare inputs of the conversions below (subnormal, tiny or non-finite),
// out of line so the common path stays short.
__device__ __noinline__ double ff_to_f64_rare(float hi, float lo) { return ff_to_f64(ff{hi, lo}); }

// hi + lo as a double for a normalised pair (|lo| <= ulp(hi) / 2), nearest
// to within half a double ulp.  lo is scaled exactly (by a power of two) into
// units of the ulp of hi widened to a double, rounded to an integer q
// (|q| <= 2^28, so it never carries out of hi's binade) and added to hi's
// widened bit pattern.  Just below a power of two the ulp halves, so a
// negative q counts twice there.  A zero pair gives a zero of hi's sign;
// subnormal, tiny (below 2^-74) and non-finite hi take ff_to_f64.
__device__ __forceinline__ double ff_to_f64_fast(ff v) {
    const unsigned uh = __float_as_uint(v.hi);
    const unsigned exh = (uh >> 23) & 0xFFu;
    if (exh - 53u > 201u) {                                    // exh < 53 or exh == 255
        if ((uh << 1) == 0u) return __longlong_as_double((long long)((unsigned long long)(uh >> 31) << 63));
        return ff_to_f64_rare(v.hi, v.lo);
    }
    const float sc = __uint_as_float((306u - exh) << 23);    // 2^(179 - exh): one ulp of double(hi) -> 1
    int q = __float2int_rn(__fmul_rn(v.lo, sc));
    if (uh >> 31) q = -q;                                      // relative to hi's magnitude
    const unsigned mh = uh & 0x7FFFFFu;
    if (mh == 0 && q < 0) q *= 2;
    const unsigned long long mag =
        ((unsigned long long)(((exh + 896u) << 20) | (mh >> 3)) << 32) | ((unsigned long long)mh << 29);
    const unsigned long long bits = (mag + (unsigned long long)(long long)q) | ((unsigned long long)(uh >> 31) << 63);
    return __longlong_as_double((long long)bits);
}

// A float as a double (exact): the bits widened for a normal value, zeros
// directly, the rest (subnormal, infinite, NaN) through ff_to_f64.
__device__ __forceinline__ double f32_to_f64_fast(float x) {
    const unsigned u = __float_as_uint(x);
    const unsigned ex = (u >> 23) & 0xFFu;
    if (ex - 1u > 253u) {                                      // zero, subnormal, infinite or NaN
        if ((u << 1) == 0u) return __longlong_as_double((long long)((unsigned long long)(u >> 31) << 63));
        if (ex == 0xFFu) {
            const unsigned long long inf_nan = 0x7FF0000000000000ull | ((unsigned long long)(u & 0x7FFFFFu) << 29);
            return __longlong_as_double((long long)(inf_nan | ((unsigned long long)(u >> 31) << 63)));
        }
        return ff_to_f64_rare(x, 0.f);
    }
    const unsigned long long bits = ((unsigned long long)(u >> 31) << 63) |
                                    ((unsigned long long)(ex + 896u) << 52) | ((unsigned long long)(u & 0x7FFFFFu) << 29);
    return __longlong_as_double((long long)bits);
}

// 1 / D for an int64 D > 0 as a normalised pair within about 2^-46 relative:
// an approximate reciprocal r, then r (1 + e) with e = 1 - D r.
__device__ __forceinline__ ff ff_recip_i64(long long D) {
    const ff d = split_i64(D);
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(d.hi));
    const float e = __fsub_rn(__fmaf_rn(-d.hi, r, 1.0f), __fmul_rn(d.lo, r));
    return fast_two_sum(r, __fmul_rn(r, e));
}

// a * b as a double, a a pair (lo need not be normalised), b a normalised pair.
__device__ __forceinline__ double ff_mul_to_f64(ff a, ff b) {
    const float p = __fmul_rn(a.hi, b.hi);
    float e = __fmaf_rn(a.hi, b.hi, -p);
    e = __fmaf_rn(a.hi, b.lo, e);
    e = __fmaf_rn(a.lo, b.hi, e);
    return ff_to_f64_fast(fast_two_sum(p, e));
}

// (n.hi + n.lo) / D for an int64 D > 0, as a double within a few units of
// 2^-46 relative: q1 from an approximate reciprocal, then one correction from
// the exact residual.
__device__ __forceinline__ double ff_div_i64_to_f64(ff n, long long D) {
    const ff d = split_i64(D);
    float inv;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(inv) : "f"(d.hi));
    const float q1 = __fmul_rn(n.hi, inv);
    const float r0 = __fmaf_rn(-q1, d.hi, n.hi);            // exact residual of the leading quotient
    const float r = __fadd_rn(__fmaf_rn(-q1, d.lo, r0), n.lo);
    const float q2 = __fmul_rn(r, inv);
    return ff_to_f64(fast_two_sum(q1, q2));
}

}  // namespace opattr
