// Sum of 2 or 4 products of doubles in fixed point on the integer pipes:
// one component of alpha * b + beta * a with complex scalars (Eq. 1, Sec. 5)
// for double data, where GB300's FP64 pipe is too narrow for a compensated
// floating-point evaluation at memory speed.
//
// Every operand must be zero or of magnitude in [2^-480, 2^480) (no
// subnormal, infinite or NaN operand; callers test this and take another
// evaluation otherwise).  Then:
//   1. each product's significand product is formed from the two 53-bit
//      significands, shifted to the top of 64 bits, by one 64 x 64 -> high
//      64 multiply: its top 64 bits (the truncated part is below 2^-62 of
//      the product);
//   2. the products are aligned to the largest exponent, 3 bits of headroom
//      added, and summed exactly as signed 64-bit integers in units
//      U = 2^-7 ulp(M) or finer (M the largest product): each alignment
//      truncates less than one U;
//   3. the integer sum is rounded once to double, to nearest even.
// The result is within 0.5 ulp(x) + n U of the exact sum x of the n exact
// products: n U <= 2^-5 ulp(M), so at most 0.5 ulp(x) + 0.032 ulp(M).  All
// intermediate magnitudes stay in the normal range: a product lies in
// [2^-960, 2^960), the sum below 2^962, and a nonzero result is a multiple of
// U >= 2^-1019.
//
// The same code compiles for the host (costa_debug_fxdot uses it), so the
// arithmetic can be checked without a GPU.
#pragma once

#include <cstdint>
#include <cstring>

#ifdef __CUDACC__
#define COSTA_FX_HD __host__ __device__ __forceinline__
#else
#define COSTA_FX_HD inline
#endif

namespace costa {
namespace fx {

COSTA_FX_HD uint64_t bits_of(double v) {
#ifdef __CUDA_ARCH__
    return static_cast<uint64_t>(__double_as_longlong(v));
#else
    uint64_t u;
    std::memcpy(&u, &v, sizeof u);
    return u;
#endif
}

COSTA_FX_HD double from_bits(uint64_t u) {
#ifdef __CUDA_ARCH__
    return __longlong_as_double(static_cast<long long>(u));
#else
    double v;
    std::memcpy(&v, &u, sizeof v);
    return v;
#endif
}

COSTA_FX_HD uint64_t mulhi(uint64_t a, uint64_t b) {
#ifdef __CUDA_ARCH__
    return __umul64hi(a, b);
#else
    return static_cast<uint64_t>((static_cast<unsigned __int128>(a) * b) >> 64);
#endif
}

COSTA_FX_HD int clz64(uint64_t v) {  // v != 0
#ifdef __CUDA_ARCH__
    return __clzll(static_cast<long long>(v));
#else
    return __builtin_clzll(v);
#endif
}

// An operand: its 53-bit significand shifted left by 11 (in [2^63, 2^64);
// 0 for a zero), its biased exponent and its sign bit.
struct Op {
    uint64_t m;
    uint32_t e;
    uint32_t s;
};

// Zero, or a magnitude in [2^-480, 2^480): the range in which unpack and
// sum below are exact as stated.
COSTA_FX_HD bool in_range(double v) {
    const uint64_t u = bits_of(v);
    const uint32_t e = static_cast<uint32_t>(u >> 52) & 0x7FFu;
    return (u << 1) == 0 || (e - (1023u - 480u)) < 960u;
}

COSTA_FX_HD Op unpack(double v) {
    const uint64_t u = bits_of(v);
    Op o;
    o.s = static_cast<uint32_t>(u >> 63);
    o.e = static_cast<uint32_t>(u >> 52) & 0x7FFu;
    o.m = o.e ? ((u << 11) | (uint64_t(1) << 63)) : 0;
    return o;
}

// One product x * y, negated when neg = 1: the top 64 bits of the
// significand product (in [2^62, 2^64), or 0), the sum of the biased
// exponents (0 for a zero product) and the sign.
struct Term {
    uint64_t p;
    uint32_t e;
    uint32_t s;
};

COSTA_FX_HD Term mul(const Op &x, const Op &y, uint32_t neg) {
    Term t;
    t.p = mulhi(x.m, y.m);
    t.e = t.p ? x.e + y.e : 0u;
    t.s = x.s ^ y.s ^ neg;
    return t;
}

// The sum of n terms, rounded once to double (to nearest, ties to even).
// A zero sum gives +0.
template <int N>
COSTA_FX_HD double sum(const Term (&t)[N]) {
    uint32_t emax = t[0].e;
#pragma unroll
    for (int i = 1; i < N; ++i) emax = t[i].e > emax ? t[i].e : emax;
    int64_t acc = 0;
#pragma unroll
    for (int i = 0; i < N; ++i) {
        const uint32_t sh = emax - t[i].e + 3u;  // >= 3: |each| < 2^61, |sum| < 2^63
        const int64_t v = sh < 64u ? static_cast<int64_t>(t[i].p >> sh) : 0;
        acc += t[i].s ? -v : v;
    }
    if (acc == 0) return 0.0;
    const uint64_t sign = acc < 0 ? uint64_t(1) << 63 : 0;
    const uint64_t mag = acc < 0 ? uint64_t(0) - static_cast<uint64_t>(acc) : static_cast<uint64_t>(acc);
    int nb = 64 - clz64(mag);  // bit length, <= 63
    uint64_t sig;
    if (nb <= 53) {
        sig = mag << (53 - nb);
    } else {
        const int sh = nb - 53;
        sig = mag >> sh;
        const uint64_t rem = mag & ((uint64_t(1) << sh) - 1), half = uint64_t(1) << (sh - 1);
        if (rem > half || (rem == half && (sig & 1))) {
            ++sig;
            if (sig >> 53) {
                sig >>= 1;
                ++nb;
            }
        }
    }
    // the acc's unit is 2^(emax - 2105); a significand of 53 bits then has
    // biased exponent nb + emax - 1083, in [4, 1985] for in-range operands
    const uint64_t be = static_cast<uint64_t>(nb) + emax - 1083u;
    return from_bits(sign | (be << 52) | (sig & ((uint64_t(1) << 52) - 1)));
}

}  // namespace fx
}  // namespace costa
