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
//
// reduce_k: for a k-bit q (2^(k-1) < q < 2^k) and x < 2^(k+63), with
//   A  = floor(x / 2^(k-1))       (below 2^64)
//   mk = floor(2^(k+63) / q)      (below 2^64, since q > 2^(k-1)),
// qe = floor(A * mk / 2^64) satisfies x/q - 2 < qe <= x/q: writing
// A = x/2^(k-1) - e1 and mk = 2^(k+63)/q - e2 with 0 <= e1, e2 < 1,
//   x/q - A*mk/2^64 <= e1 * 2^(k-1)/q + e2 * x/2^(k+63) < 1 + 1,
// so r = x - qe*q lies in [0, 3q): two conditional subtractions.  One
// 64x64 high product replaces the five partial products of reduce128.
#pragma once
#include <stdint.h>

struct LimbConst {
    uint64_t q;
    uint64_t mu_hi;
    uint64_t mu_lo;
    uint64_t mu64;
    uint64_t mk;   // floor(2^(k+63) / q), k = bit length of q (reduce_k)
    uint64_t km1;  // k - 1
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
// Narrow residues (q < 2^52): radix-2^26 split form and Karatsuba products.
//
// A residue a < 2^52 is kept as one 64-bit word whose low 32-bit half holds
// a0 = a mod 2^26 and whose high half holds a1 = floor(a / 2^26).  For two
// such residues,
//   a * b = a0*b0 + ((a0+a1)*(b0+b1) - a0*b0 - a1*b1) * 2^26 + a1*b1 * 2^52
// (Karatsuba), so a product-accumulate is three 32x32 -> 64-bit
// multiply-adds into accumulators lo, x, hi; the middle term is recovered
// once, at the reduction.  (a0+a1)*(b0+b1) < 2^54, so the accumulators hold
// any 1023 products without wrapping (kNarrowMacBudget), and the weighted sum
// stays below 2^116.
//
// Split words can also be summed as plain 64-bit integers: 64 of them keep
// each half below 2^32 (64 * (2^26 - 1) < 2^32), so a packed sum of at most
// 64 split words reads back as (sum of a0) + (sum of a1) * 2^26 < 2^59.
// ---------------------------------------------------------------------------
constexpr uint32_t kNarrowMacBudget = 1023;
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

// (lo, x, hi) += split a times split b, Karatsuba.  Each 32x32 -> 64-bit
// product is formed alone and added with a plain 64-bit add: measured on
// sm_103a this keeps the multiplier pipe (the limit here) less busy than a
// multiply-add into the 64-bit accumulator.  `z` is zero, but a value known
// only at run time (a kernel argument): the half sums a0 + a1 + z and
// b0 + b1 + z are then three-input additions, which the compiler issues on
// the integer ALU instead of as multiply-adds on the multiplier pipe
// (measured on GB300: that pipe 67% -> 59% busy on the BERT layer, the ALU
// 33% -> 41%, the layer kernels 0.5-1.5% faster).
__device__ __forceinline__ void mac26(uint64_t &lo, uint64_t &x, uint64_t &hi, uint64_t as, uint64_t bs,
                                      uint32_t z)
{
    const uint32_t a0 = (uint32_t)as, a1 = (uint32_t)(as >> 32);
    const uint32_t b0 = (uint32_t)bs, b1 = (uint32_t)(bs >> 32);
    uint64_t p0, p1, p2;
    asm("mul.wide.u32 %0, %3, %4;\n\t"
        "mul.wide.u32 %1, %5, %6;\n\t"
        "mul.wide.u32 %2, %7, %8;"
        : "=l"(p0), "=l"(p1), "=l"(p2)
        : "r"(a0), "r"(b0), "r"(a0 + a1 + z), "r"(b0 + b1 + z), "r"(a1), "r"(b1));
    lo += p0;
    x += p1;
    hi += p2;
}

// x1 * 2^64 + x0 mod q for a value below 2^(k+63) (see reduce_k above)
__device__ __forceinline__ uint64_t reduce_k(uint64_t x0, uint64_t x1, const LimbConst &m)
{
    const uint32_t s = (uint32_t)m.km1;  // 1 <= k - 1 <= 51
    const uint64_t A = (x0 >> s) | (x1 << (64 - s));
    const uint64_t qe = __umul64hi(A, m.mk);
    uint64_t r = x0 - qe * m.q;  // the true remainder is below 3q < 2^64
    r = r >= m.q ? r - m.q : r;
    return r >= m.q ? r - m.q : r;
}

// lo + (x - lo - hi) * 2^26 + hi * 2^52 mod q: the value of at most 1023
// products of residues below q < 2^52 (kNarrowMacBudget), so below
// 2^10 q^2 < 2^(2k+10) <= 2^(k+63), which reduce_k takes
__device__ __forceinline__ uint64_t reduce26(uint64_t lo, uint64_t x, uint64_t hi, const LimbConst &m)
{
    const uint64_t mid = x - lo - hi;
    uint64_t x0 = lo, x1 = 0;
    asm("add.cc.u64 %0, %0, %2;\n\t"
        "addc.u64   %1, %1, %3;\n\t"
        "add.cc.u64 %0, %0, %4;\n\t"
        "addc.u64   %1, %1, %5;"
        : "+l"(x0), "+l"(x1)
        : "l"(mid << 26), "l"(mid >> 38), "l"(hi << 52), "l"(hi >> 12));
    return reduce_k(x0, x1, m);
}

}  // namespace rns
#endif  // __CUDACC__
