// tile_math.cuh -- per-lane tile arithmetic shared by the tiled kernels:
// vectors of C coefficients per lane, shared-memory and global accessors,
// the two arithmetic policies (any q < 2^60, and radix-2^26 split words for
// q < 2^52), and lazy signed sums over runs of source tiles.
#pragma once
#include <stdint.h>

#include "rns.cuh"

namespace tile {

// The limb's constants, read from shared memory where they are needed
// (kept out of registers between uses).
__device__ __forceinline__ LimbConst load_limb(uint32_t addr)
{
    LimbConst m;
    asm volatile("ld.shared.v2.u64 {%0, %1}, [%2];" : "=l"(m.q), "=l"(m.mu_hi) : "r"(addr));
    asm volatile("ld.shared.v2.u64 {%0, %1}, [%2+16];" : "=l"(m.mu_lo), "=l"(m.mu64) : "r"(addr));
    // (not volatile: dropped where only the first four are used)
    asm("ld.shared.v2.u64 {%0, %1}, [%2+32];" : "=l"(m.mk), "=l"(m.km1) : "r"(addr));
    return m;
}

template <int C>
struct V {
    uint64_t x[C];
};

// one lane's C plaintext words, not cached in L1
template <int C>
__device__ __forceinline__ V<C> ldg_stream(const uint64_t *p, uint64_t pol)
{
    V<C> v;
    if constexpr (C == 2)
        asm("ld.global.nc.L1::no_allocate.L2::cache_hint.v2.u64 {%0, %1}, [%2], %3;"
            : "=l"(v.x[0]), "=l"(v.x[1])
            : "l"(p), "l"(pol));
    else
        asm("ld.global.nc.L1::no_allocate.L2::cache_hint.u64 %0, [%1], %2;"
            : "=l"(v.x[0])
            : "l"(p), "l"(pol));
    return v;
}

// shared memory through byte offsets from the dynamic shared array
template <int C>
__device__ __forceinline__ V<C> lds(const char *sm, uint32_t off)
{
    V<C> v;
    if constexpr (C == 2) {
        const ulonglong2 t = *reinterpret_cast<const ulonglong2 *>(sm + off);
        v.x[0] = t.x;
        v.x[1] = t.y;
    } else {
        v.x[0] = *reinterpret_cast<const uint64_t *>(sm + off);
    }
    return v;
}

template <int C>
__device__ __forceinline__ void sts(char *sm, uint32_t off, const V<C> &v)
{
    if constexpr (C == 2)
        *reinterpret_cast<ulonglong2 *>(sm + off) = make_ulonglong2(v.x[0], v.x[1]);
    else
        *reinterpret_cast<uint64_t *>(sm + off) = v.x[0];
}

template <int C>
__device__ __forceinline__ void stg(uint64_t *p, const V<C> &v)
{
    if constexpr (C == 2)
        *reinterpret_cast<ulonglong2 *>(p) = make_ulonglong2(v.x[0], v.x[1]);
    else
        *p = v.x[0];
}

// ---------------------------------------------------------------------------
// Arithmetic policies.  "Operand form" is how source residues sit in shared
// memory: canonical for Wide, split for Narrow.
// ---------------------------------------------------------------------------
template <bool NARROW>
struct Arith;

// Any q < 2^60: 128-bit products (lo, hi), plain 64-bit sums.
template <>
struct Arith<false> {
    struct Acc {
        uint64_t lo, hi;
    };
    __device__ static uint64_t operand(uint64_t a) { return a; }
    __device__ static void zero(Acc &a) { a.lo = a.hi = 0; }
    __device__ static void mac(Acc &a, uint64_t x, uint64_t y, uint32_t /*zero*/ = 0) { rns::mac(a.lo, a.hi, x, y); }
    __device__ static uint64_t reduce(const Acc &a, const LimbConst &m) { return rns::reduce128(a.lo, a.hi, m); }
    __device__ static void fold(Acc &a, const LimbConst &m)
    {
        a.lo = reduce(a, m);
        a.hi = 0;
    }
    // canonical residue of P - M, each a plain sum within the lazy-sum bound
    __device__ static uint64_t signed_value(uint64_t p, uint64_t mm, const LimbConst &m)
    {
        return rns::sub_mod(rns::reduce64(p, m), rns::reduce64(mm, m), m.q);
    }
    // the same for narrow moduli (q < 2^52): P and M are sums of at most 64
    // run terms and six slot terms, each below q, so P + 128q - M is positive
    // and below 2^60: one reduction
    __device__ static uint64_t signed_value_narrow(uint64_t p, uint64_t mm, const LimbConst &m)
    {
        return rns::reduce64(p + 128 * m.q - mm, m);
    }
};

// q < 2^52: every factor in split form (sources split in shared memory or
// where a product reads them, the other factor split on the way in);
// Karatsuba products into three accumulators; packed sums of split words.
template <>
struct Arith<true> {
    struct Acc {
        uint64_t lo, x, hi;
    };
    __device__ static uint64_t operand(uint64_t a) { return rns::split26(a); }
    __device__ static void zero(Acc &a) { a.lo = a.x = a.hi = 0; }
    // both factors in operand (split) form; `zero` as in rns::mac26 (a
    // literal 0 folds the half sums back into two-input additions)
    __device__ static void mac(Acc &a, uint64_t x, uint64_t y, uint32_t zero = 0)
    {
        rns::mac26(a.lo, a.x, a.hi, x, y, zero);
    }
    __device__ static uint64_t reduce(const Acc &a, const LimbConst &m) { return rns::reduce26(a.lo, a.x, a.hi, m); }
    __device__ static void fold(Acc &a, const LimbConst &m)
    {
        a.lo = reduce(a, m);
        a.x = a.lo;  // the middle term x - lo - hi stays 0
        a.hi = 0;
    }
    // P - M + 64q is below 2^59 (each packed sum reads back below 2^58)
    __device__ static uint64_t signed_value(uint64_t p, uint64_t mm, const LimbConst &m)
    {
        const uint64_t k = (uint64_t)rns::kNarrowSumBudget * m.q;
        return rns::reduce64(rns::unsplit_sum(p) + k - rns::unsplit_sum(mm), m);
    }
};

// Sum of the n source tiles (both polys) named by the 16-bit indices packed
// two per word from schedule byte offset `wp`; `src` = this lane's offset in
// the source region.  K indices per step (each decoded once, its two polys
// read at offsets 0 and TB), their loads independent, and the next step's
// index words requested before this step's additions (the last request may
// read words past the run: they lie inside the dynamic shared memory, which
// continues with the source region, and are not used).  Returns the offset
// just past the run's words.
template <int C, uint32_t TB>
__device__ __forceinline__ uint32_t run_sum(const char *sm, uint32_t src, uint32_t wp, uint32_t n, V<C> &s0,
                                            V<C> &s1)
{
    constexpr uint32_t PB = 2 * TB;
    constexpr uint32_t K = C == 1 ? 8 : 2;  // 2K loads of C words in flight
    constexpr uint32_t NW = K / 2;          // index words per step
    uint32_t k = 0;
    if (n >= K) {
        uint32_t w[NW];
#pragma unroll
        for (uint32_t j = 0; j < NW; ++j) w[j] = *reinterpret_cast<const uint32_t *>(sm + wp + 4 * j);
        for (; k + K <= n; k += K, wp += 4 * NW) {
            V<C> a[K], b[K];
#pragma unroll
            for (uint32_t j = 0; j < K; ++j) {
                const uint32_t o = src + ((j & 1) ? (w[j / 2] >> 16) : (w[j / 2] & 0xffffu)) * PB;
                a[j] = lds<C>(sm, o);
                b[j] = lds<C>(sm, o + TB);
            }
#pragma unroll
            for (uint32_t j = 0; j < NW; ++j) w[j] = *reinterpret_cast<const uint32_t *>(sm + wp + 4 * NW + 4 * j);
#pragma unroll
            for (int x = 0; x < C; ++x) {
#pragma unroll
                for (uint32_t j = 0; j + 1 < K; j += 2) {  // three-input additions
                    s0.x[x] = s0.x[x] + a[j].x[x] + a[j + 1].x[x];
                    s1.x[x] = s1.x[x] + b[j].x[x] + b[j + 1].x[x];
                }
            }
        }
    }
    for (; k + 2 <= n; k += 2, wp += 4) {
        const uint32_t w = *reinterpret_cast<const uint32_t *>(sm + wp);
        const uint32_t o0 = src + (w & 0xffffu) * PB, o1 = src + (w >> 16) * PB;
        const V<C> a0 = lds<C>(sm, o0), a1 = lds<C>(sm, o1), b0 = lds<C>(sm, o0 + TB), b1 = lds<C>(sm, o1 + TB);
#pragma unroll
        for (int x = 0; x < C; ++x) {
            s0.x[x] += a0.x[x] + a1.x[x];
            s1.x[x] += b0.x[x] + b1.x[x];
        }
    }
    if (k < n) {
        const uint32_t w = *reinterpret_cast<const uint32_t *>(sm + wp);
        const uint32_t o0 = src + (w & 0xffffu) * PB;
        const V<C> a0 = lds<C>(sm, o0), b0 = lds<C>(sm, o0 + TB);
#pragma unroll
        for (int x = 0; x < C; ++x) {
            s0.x[x] += a0.x[x];
            s1.x[x] += b0.x[x];
        }
        wp += 4;
    }
    return wp;
}

// The same sum over a run of byte offsets (one 32-bit word per source: the
// source's offset from the start of the region, so that its address is one
// addition), the run starting on a 16-byte boundary and padded to a multiple
// of four words.  K offsets per step, read with one vector load, the
// next step's requested before this step's additions (that request may read
// words past the run, inside the dynamic shared memory as above, unused).
// Returns the offset just past the padded run.
template <int C, uint32_t TB>
__device__ __forceinline__ uint32_t run_sum_offsets(const char *sm, uint32_t src, uint32_t wp, uint32_t n, V<C> &s0,
                                                    V<C> &s1)
{
    // 2K loads of C words in flight (measured on GB300 with one coefficient
    // per lane: VGG 2.307 ms with K = 8, 2.274 ms with 4; with two, 2 beats 4)
    constexpr uint32_t K = C == 1 ? 4 : 2;
    uint32_t k = 0;
    if (n >= K) {
        uint32_t o[K];
        auto get = [&](uint32_t at) {
            if constexpr (K == 4) {
                const uint4 x = *reinterpret_cast<const uint4 *>(sm + at);
                o[0] = x.x, o[1] = x.y, o[2] = x.z, o[3] = x.w;
            } else {
                const uint2 x = *reinterpret_cast<const uint2 *>(sm + at);
                o[0] = x.x, o[1] = x.y;
            }
        };
        get(wp);
        for (; k + K <= n; k += K, wp += 4 * K) {
            V<C> a[K], b[K];
#pragma unroll
            for (uint32_t j = 0; j < K; ++j) {
                a[j] = lds<C>(sm, src + o[j]);
                b[j] = lds<C>(sm, src + o[j] + TB);
            }
            get(wp + 4 * K);
#pragma unroll
            for (int x = 0; x < C; ++x) {
#pragma unroll
                for (uint32_t j = 0; j + 1 < K; j += 2) {  // three-input additions
                    s0.x[x] = s0.x[x] + a[j].x[x] + a[j + 1].x[x];
                    s1.x[x] = s1.x[x] + b[j].x[x] + b[j + 1].x[x];
                }
            }
        }
    }
    for (; k + 2 <= n; k += 2, wp += 8) {
        const uint2 w = *reinterpret_cast<const uint2 *>(sm + wp);
        const V<C> a0 = lds<C>(sm, src + w.x), a1 = lds<C>(sm, src + w.y);
        const V<C> b0 = lds<C>(sm, src + w.x + TB), b1 = lds<C>(sm, src + w.y + TB);
#pragma unroll
        for (int x = 0; x < C; ++x) {
            s0.x[x] += a0.x[x] + a1.x[x];
            s1.x[x] += b0.x[x] + b1.x[x];
        }
    }
    if (k < n) {
        const uint32_t o0 = src + *reinterpret_cast<const uint32_t *>(sm + wp);
        const V<C> a0 = lds<C>(sm, o0), b0 = lds<C>(sm, o0 + TB);
#pragma unroll
        for (int x = 0; x < C; ++x) {
            s0.x[x] += a0.x[x];
            s1.x[x] += b0.x[x];
        }
        wp += 4;
    }
    return (wp + 15) & ~15u;  // the run started on a 16-byte boundary
}

// Signed sum of the program at byte offset `hdr`, both polys, as canonical
// residues; SPLIT: the sources are in split form (else canonical, whatever
// the arithmetic).  A program starts with n_plus | n_minus << 16.  In the
// packed form (`offsets` false) the plus run and the minus run of 16-bit
// source indices follow, then one slot word: n_plus_slots | n_minus_slots
// << 4 and up to six 4-bit slot numbers from bit 8 (plus slots first).  In
// the offset form the slot word is the second word, the program's first four
// words are a block of their own (the third holds a formation's target slot),
// and each run is a run of source byte offsets padded to four words
// (run_sum_offsets); every offset-form program starts on a 16-byte boundary.
// A slot is a tile pair of this warp's slot area at byte offset `slots`
// (this lane's words of slot 0), holding a shared signed sum the warp formed
// earlier.  Returns the offset just past the program.
// NC: canonical sources with narrow moduli (Arith<false>::signed_value_narrow).
template <bool SPLIT, int C, uint32_t TB, bool NC = false>
__device__ __forceinline__ uint32_t signed_sum(const char *sm, uint32_t src, uint32_t hdr, uint32_t lim,
                                               uint32_t slots, V<C> &o0, V<C> &o1, bool offsets = false)
{
    using A = Arith<SPLIT>;
    constexpr uint32_t PB = 2 * TB;
    const uint32_t h = *reinterpret_cast<const uint32_t *>(sm + hdr);
    V<C> p0{}, p1{}, m0{}, m1{};
    uint32_t next, sw;
    if (offsets) {
        sw = *reinterpret_cast<const uint32_t *>(sm + hdr + 4);
        next = run_sum_offsets<C, TB>(sm, src, hdr + 16, h & 0xffffu, p0, p1);
        next = run_sum_offsets<C, TB>(sm, src, next, h >> 16, m0, m1);
    } else {
        uint32_t wp = run_sum<C, TB>(sm, src, hdr + 4, h & 0xffffu, p0, p1);
        wp = run_sum<C, TB>(sm, src, wp, h >> 16, m0, m1);
        sw = *reinterpret_cast<const uint32_t *>(sm + wp);
        next = wp + 4;
    }
    const uint32_t nps = sw & 15u, ns = nps + ((sw >> 4) & 15u);
    for (uint32_t j = 0; j < ns; ++j) {
        const uint32_t o = slots + ((sw >> (8 + 4 * j)) & 15u) * PB;
        const V<C> a = lds<C>(sm, o), b = lds<C>(sm, o + TB);
        V<C> &t0 = j < nps ? p0 : m0;
        V<C> &t1 = j < nps ? p1 : m1;
#pragma unroll
        for (int x = 0; x < C; ++x) {
            t0.x[x] += a.x[x];
            t1.x[x] += b.x[x];
        }
    }
    const LimbConst m = load_limb(lim);
#pragma unroll
    for (int x = 0; x < C; ++x) {
        if constexpr (NC && !SPLIT) {
            o0.x[x] = Arith<false>::signed_value_narrow(p0.x[x], m0.x[x], m);
            o1.x[x] = Arith<false>::signed_value_narrow(p1.x[x], m1.x[x], m);
        } else {
            o0.x[x] = A::signed_value(p0.x[x], m0.x[x], m);
            o1.x[x] = A::signed_value(p1.x[x], m1.x[x], m);
        }
    }
    return next;
}

}  // namespace tile
