// rns.cuh -- RNS modular-arithmetic core for residues of primes q < 2^60.
//
// Residues are canonical uint64 values in [0, q).  Products of two residues
// are < 2^120 and are accumulated lazily in 128 bits (lo, hi); the host
// bounds how many products may be added before a reduction (at least 256 for
// q < 2^60).  Reductions use Barrett's method with constants computed on the
// host per limb:
//
//   mu   = floor(2^128 / q)   (two words: mu_hi, mu_lo)
//   mu64 = floor(2^64  / q)
//
// reduce128: for x < 2^128, qe = floor(x * mu / 2^128) satisfies
//   x/q - 1 < x*mu/2^128 <= x/q,
// so qe is floor(x/q) or floor(x/q) - 1 and r = x - qe*q lies in [0, 2q);
// one conditional subtraction gives the canonical residue.  Only the low 64
// bits of qe are needed, because r < 2^64.  Writing x = x1*2^64 + x0 and
// mu = mu1*2^64 + mu0,
//   floor(x*mu / 2^128) = x1*mu1 + floor((x1*mu0 + x0*mu1 + hi(x0*mu0)) / 2^64),
// since the dropped low word of x0*mu0 is below 2^64 and cannot carry.
//
// reduce64: for x < 2^64, qe = hi(x * mu64) is floor(x/q) or one less, the
// same argument with 2^64 in place of 2^128.
#pragma once
#include <stdint.h>

struct LimbConst {
    uint64_t q;
    uint64_t mu_hi;
    uint64_t mu_lo;
    uint64_t mu64;
};

#if defined(__CUDACC__)
namespace rns {

// acc (lo, hi) += a * b, full 128-bit product, carry chained.
__device__ __forceinline__ void mac(uint64_t &lo, uint64_t &hi, uint64_t a, uint64_t b)
{
    asm("mad.lo.cc.u64 %0, %2, %3, %0;\n\t"
        "madc.hi.u64   %1, %2, %3, %1;"
        : "+l"(lo), "+l"(hi)
        : "l"(a), "l"(b));
}

// (lo, hi) = a * b
__device__ __forceinline__ void mul_wide(uint64_t &lo, uint64_t &hi, uint64_t a, uint64_t b)
{
    lo = a * b;
    hi = __umul64hi(a, b);
}

// (lo, hi) += x (64-bit)
__device__ __forceinline__ void add_wide(uint64_t &lo, uint64_t &hi, uint64_t x)
{
    asm("add.cc.u64 %0, %0, %2;\n\t"
        "addc.u64   %1, %1, 0;"
        : "+l"(lo), "+l"(hi)
        : "l"(x));
}

__device__ __forceinline__ uint64_t reduce128(uint64_t x0, uint64_t x1, const LimbConst &m)
{
    const uint64_t a_lo = x0 * m.mu_hi, a_hi = __umul64hi(x0, m.mu_hi);
    const uint64_t b_lo = x1 * m.mu_lo, b_hi = __umul64hi(x1, m.mu_lo);
    const uint64_t c = __umul64hi(x0, m.mu_lo);
    // t = a + b + c (130 bits); only its middle word tmid = floor(t/2^64) mod 2^64
    uint64_t s, tmid;
    asm("add.cc.u64  %0, %2, %3;\n\t"
        "addc.u64    %1, %4, %5;"
        : "=l"(s), "=l"(tmid)
        : "l"(a_lo), "l"(b_lo), "l"(a_hi), "l"(b_hi));
    asm("add.cc.u64  %0, %0, %2;\n\t"
        "addc.u64    %1, %1, 0;"
        : "+l"(s), "+l"(tmid)
        : "l"(c));
    const uint64_t qe = x1 * m.mu_hi + tmid;
    uint64_t r = x0 - qe * m.q;
    return r >= m.q ? r - m.q : r;
}

__device__ __forceinline__ uint64_t reduce64(uint64_t x, const LimbConst &m)
{
    const uint64_t qe = __umul64hi(x, m.mu64);
    const uint64_t r = x - qe * m.q;
    return r >= m.q ? r - m.q : r;
}

__device__ __forceinline__ uint64_t add_mod(uint64_t a, uint64_t b, uint64_t q)
{
    const uint64_t s = a + b;  // a, b < q < 2^60: no wrap
    return s >= q ? s - q : s;
}

__device__ __forceinline__ uint64_t sub_mod(uint64_t a, uint64_t b, uint64_t q)
{
    return a >= b ? a - b : a + (q - b);
}

}  // namespace rns
#endif  // __CUDACC__
