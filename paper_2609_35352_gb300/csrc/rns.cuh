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

// ---------------------------------------------------------------------------
// Narrow residues (q < 2^52): one operand in radix-2^26 split form.
//
// A residue a < 2^52 is kept as one 64-bit word whose low 32-bit half holds
// a0 = a mod 2^26 and whose high half holds a1 = floor(a / 2^26).  The other
// factor b is any 64-bit value below 2^59, taken as b = b1 * 2^32 + b0.  Then
//   a * b = a0*b0 + a1*b0 * 2^26 + a0*b1 * 2^32 + a1*b1 * 2^58,
// four 32x32 -> 64-bit multiply-adds into four 64-bit accumulators.  The
// first two grow by less than 2^58 per product and the last two by less
// than 2^53, so the accumulators hold any 64 products without wrapping
// (kNarrowMacBudget), and their weighted sum stays below 2^118.
//
// Split words can also be summed as plain 64-bit integers: 64 of them keep
// each half below 2^32 (64 * (2^26 - 1) < 2^32), so a packed sum of at most
// 64 split words reads back as (sum of a0) + (sum of a1) * 2^26 < 2^59.
// ---------------------------------------------------------------------------
constexpr uint32_t kNarrowMacBudget = 64;
constexpr uint32_t kNarrowSumBudget = 64;

__device__ __forceinline__ uint64_t split26(uint64_t a)
{
    const uint32_t lo = (uint32_t)a & 0x3FFFFFFu;
    const uint32_t hi = (uint32_t)(a >> 26);
    return ((uint64_t)hi << 32) | lo;
}

// value of a packed sum of at most kNarrowSumBudget split words (< 2^59)
__device__ __forceinline__ uint64_t unsplit_sum(uint64_t w)
{
    return (w & 0xFFFFFFFFull) + ((w >> 32) << 26);
}

// (a00, a10, a01, a11) += split a times b (b < 2^59)
__device__ __forceinline__ void mac26(uint64_t &a00, uint64_t &a10, uint64_t &a01, uint64_t &a11,
                                      uint64_t as, uint64_t b)
{
    const uint32_t x0 = (uint32_t)as, x1 = (uint32_t)(as >> 32);
    const uint32_t y0 = (uint32_t)b, y1 = (uint32_t)(b >> 32);
    asm("mad.wide.u32 %0, %4, %6, %0;\n\t"
        "mad.wide.u32 %1, %5, %6, %1;\n\t"
        "mad.wide.u32 %2, %4, %7, %2;\n\t"
        "mad.wide.u32 %3, %5, %7, %3;"
        : "+l"(a00), "+l"(a10), "+l"(a01), "+l"(a11)
        : "r"(x0), "r"(x1), "r"(y0), "r"(y1));
}

// a00 + a10 * 2^26 + a01 * 2^32 + a11 * 2^58 mod q (the sum is below 2^118)
__device__ __forceinline__ uint64_t reduce26(uint64_t a00, uint64_t a10, uint64_t a01, uint64_t a11,
                                             const LimbConst &m)
{
    uint64_t x0 = a00, x1 = 0;
    asm("add.cc.u64 %0, %0, %2;\n\t"
        "addc.u64   %1, %1, %3;\n\t"
        "add.cc.u64 %0, %0, %4;\n\t"
        "addc.u64   %1, %1, %5;\n\t"
        "add.cc.u64 %0, %0, %6;\n\t"
        "addc.u64   %1, %1, %7;"
        : "+l"(x0), "+l"(x1)
        : "l"(a10 << 26), "l"(a10 >> 38), "l"(a01 << 32), "l"(a01 >> 32), "l"(a11 << 58),
          "l"(a11 >> 6));
    return reduce128(x0, x1, m);
}

}  // namespace rns
#endif  // __CUDACC__
