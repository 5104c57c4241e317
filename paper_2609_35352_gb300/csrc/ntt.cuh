// ntt.cuh -- the negacyclic transform machinery shared by the rescale
// (rescale.cu) and the plaintext encoder (encode.cu).
//
// Transform.  For a poly a of N = 2^n coefficients and psi a primitive 2N-th
// root of unity, the forward transform is A[k] = a(psi^(2 brv(k) + 1)),
// brv reversing the n bits of k: the radix-2 Cooley-Tukey stages (at the
// stage with m blocks, block i pairs elements at distance N / 2m with
// twiddle psi^brv(m + i)) from natural to bit-reversed order.  The inverse
// runs the Gentleman-Sande stages in the opposite order with psi^-brv(m + i)
// and then multiplies by N^-1.  The same stages serve residues mod q (psi a
// root mod q; the NTT of the RNS limbs) and complex numbers (psi =
// exp(i pi / N); the canonical embedding of CKKS, whose slots are values of
// the plaintext at odd powers of psi).
//
// Passes.  The stages are split between two passes over memory (N = R1 * R2,
// R1 = 2^floor(n/2)):
//   high pass  the first log2(R1) stages: for a fixed low index, the R1
//              elements hi * R2 + lo form one sub-transform; a CTA takes
//              tile / R1 of them (adjacent columns, so accesses coalesce);
//   low pass   the other stages, inside blocks of R2 consecutive elements;
//              a CTA takes tile / R2 blocks.
// A CTA's tile is 4096 elements in the high pass and 2048 in the low pass
// (whose CTAs also stage about one twiddle per element: the smaller tile lets
// more CTAs share an SM); a thread handles 16 elements.
// A pass runs its stages in rounds of up to 4: in a round each thread holds
// the 2^K elements of one group in registers, spaced by the round's smallest
// distance, and applies the round's K stages to them (a group needs 2^K - 1
// twiddles).  Rounds hand over through shared memory ([sub-transform]
// [position], one element of padding per row against bank conflicts); the
// first and last rounds of a pass read and write global memory directly
// wherever their access pattern coalesces.  The CTA's twiddles are copied to
// shared memory (cp.async) while its data loads are in flight.  Everything is
// instantiated per log2 N, so all index arithmetic is constant-folded.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace fiona_ntt {

constexpr int kLogTileMax = 12;  // at most 4096 elements per CTA (2048 in the low pass)
constexpr int kLogNMin = 10, kLogNMax = 17;  // the ring dimensions a context accepts

// ---------------------------------------------------------------------------
// Residues mod q < 2^60 in 64-bit words.  A product by a table constant w
// uses Shoup's precomputed w' = floor(w 2^64 / q): r = x w - floor(x w' /
// 2^64) q lies in [0, 2q) for any 64-bit x.  The quotient is taken from
// three of the four 32-bit partial products of x w' (the low-by-low one and
// the carries below bit 64 are dropped), which underestimates it by at most
// 2, so r lies in [0, 4q).
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t mul_shoup_lazy(uint64_t x, ulonglong2 w, uint64_t q)
{
    const uint32_t xl = (uint32_t)x, xh = (uint32_t)(x >> 32);
    const uint32_t wl = (uint32_t)w.y, wh = (uint32_t)(w.y >> 32);
    const uint64_t qh = (uint64_t)xh * wh + __umulhi(xh, wl) + __umulhi(xl, wh);
    return x * w.x + qh * (0 - q);
}

__device__ __forceinline__ uint64_t csub(uint64_t x, uint64_t c) { return x >= c ? x - c : x; }

// x in [0, 4q) -> canonical
__device__ __forceinline__ uint64_t canon4(uint64_t x, uint64_t q) { return csub(csub(x, 2 * q), q); }

// x mod q for any 64-bit x: floor(x * mu64 / 2^64), mu64 = floor(2^64 / q),
// is floor(x / q) or one less
__device__ __forceinline__ uint64_t reduce_any(uint64_t x, uint64_t q, uint64_t mu64)
{
    return csub(x - __umul64hi(x, mu64) * q, q);
}

// Modular butterflies.  Values between stages:
//   forward, general   in [0, 8q): x is brought below 4q before each
//                      butterfly (x + t, x - t + 4q with t in [0, 4q));
//   forward, FAST      (q < 2^56, inputs below 5q) no reduction at all: each
//                      stage adds less than 4q to the bound, so after at most
//                      17 stages values stay below 73q < 2^63;
//   inverse            in [0, 4q): x + y is brought below 4q, and
//                      x - y + 4q is only multiplied.
template <bool FAST>
struct ModArith {
    typedef uint64_t T;
    typedef ulonglong2 W;  // (w, Shoup companion)
    uint64_t q;
    __device__ __forceinline__ void ct(T &x, T &y, W w) const
    {
        const uint64_t a = FAST ? x : csub(x, 4 * q);
        const uint64_t t = mul_shoup_lazy(y, w, q);
        x = a + t;
        y = a + 4 * q - t;
    }
    __device__ __forceinline__ void gs(T &x, T &y, W w) const
    {
        const uint64_t a = x, b = y;
        x = csub(a + b, 4 * q);
        y = mul_shoup_lazy(a + 4 * q - b, w, q);
    }
};

// Complex numbers in fp64 (re, im); twiddles are (cos, sin) pairs.
struct CplxArith {
    typedef double2 T;
    typedef double2 W;
    __device__ __forceinline__ static double2 mul(double2 a, double2 b)
    {
        return make_double2(fma(a.x, b.x, -a.y * b.y), fma(a.x, b.y, a.y * b.x));
    }
    __device__ __forceinline__ void ct(T &x, T &y, W w) const
    {
        const double2 t = mul(y, w);
        y = make_double2(x.x - t.x, x.y - t.y);
        x = make_double2(x.x + t.x, x.y + t.y);
    }
    __device__ __forceinline__ void gs(T &x, T &y, W w) const
    {
        const double2 d = make_double2(x.x - y.x, x.y - y.y);
        x = make_double2(x.x + y.x, x.y + y.y);
        y = mul(d, w);
    }
};

// ---------------------------------------------------------------------------
// Compile-time geometry
// ---------------------------------------------------------------------------
template <int LOGN>
struct Shape {
    static constexpr int n1 = LOGN / 2;
    static constexpr int lt = LOGN < kLogTileMax ? LOGN : kLogTileMax;  // log2(tile)
    static constexpr int ltiles = LOGN - lt;                            // log2(tiles per transform)
};

// A pass over a tile: 2^LSUBS sub-transforms of 2^S positions, in rounds,
// 2^LTILES tiles per transform, 16 elements per thread (at least 64 threads).
template <int S, int LSUBS, bool HIGH, int LTILES>
struct PassShape {
    static constexpr int s = S, lsubs = LSUBS, subs = 1 << LSUBS;
    static constexpr int tile = 1 << (S + LSUBS);
    static constexpr int ltiles = LTILES;
    static constexpr uint32_t threads = tile / 16 < 64 ? 64 : tile / 16;
    static constexpr int pitch = (1 << S) + 1;
    static constexpr int nr = (S + 3) / 4;
    __host__ __device__ static constexpr int K(int r) { return S / nr + (r < S % nr ? 1 : 0); }
    __host__ __device__ static constexpr int J0(int r) { return r == 0 ? 0 : J0(r - 1) + K(r - 1); }
    static constexpr bool high = HIGH;
    // shared memory: the staged twiddles (2^s entries for the high pass, at
    // most one per tile element for the low pass), then the padded tile
    static constexpr int tw_entries = HIGH ? 1 << S : 1 << (S + LSUBS);
    template <class A>
    __host__ __device__ static constexpr size_t smem_bytes()
    {
        return sizeof(typename A::W) * tw_entries + sizeof(typename A::T) * subs * pitch;
    }
};

template <int LOGN>
using HighPass = PassShape<Shape<LOGN>::n1, Shape<LOGN>::lt - Shape<LOGN>::n1, true, Shape<LOGN>::ltiles>;
// the low pass: a tile of half the high pass's, but at least one block
template <int LOGN>
struct LowShape {
    static constexpr int s = LOGN - Shape<LOGN>::n1;
    static constexpr int lt = Shape<LOGN>::lt - 1 > s ? Shape<LOGN>::lt - 1 : s;
};
template <int LOGN>
using LowPass = PassShape<LowShape<LOGN>::s, LowShape<LOGN>::lt - LowShape<LOGN>::s, false, LOGN - LowShape<LOGN>::lt>;

// Group g of round R: sub-transform `sub`, and the element positions
// (hi << (lD + K)) + (i << lD) + lo, i < 2^K.  High pass: sub-transforms
// fastest (adjacent columns); low pass: lo fastest (adjacent elements).
template <class PS, int R>
struct Group {
    static constexpr int K = PS::K(R), J0 = PS::J0(R), LD = PS::s - J0 - K;
    static constexpr int groups = PS::tile >> K;
    static constexpr int per_thread = (groups + (int)PS::threads - 1) / (int)PS::threads;
    uint32_t sub, hi, lo;
    __device__ __forceinline__ explicit Group(uint32_t g)
    {
        if (PS::high) {
            sub = g & (PS::subs - 1);
            const uint32_t rest = g >> PS::lsubs;
            lo = rest & ((1u << LD) - 1);
            hi = rest >> LD;
        } else {
            lo = g & ((1u << LD) - 1);
            const uint32_t rest = g >> LD;
            sub = rest & (PS::subs - 1);
            hi = rest >> PS::lsubs;
        }
    }
    __device__ __forceinline__ uint32_t pos(int i) const { return (hi << (LD + K)) + ((uint32_t)i << LD) + lo; }
    // twiddle of local stage J0 + k, block b of the group, in the staged layout
    __device__ __forceinline__ uint32_t tw(int k, int b) const
    {
        const int j = J0 + k;
        if (PS::high) return (1u << j) + (hi << k) + b;
        return ((PS::subs << j) - PS::subs) + (((hi << k) + b) << PS::lsubs) + sub;
    }
};

template <class PS, int R, int k, bool INV, class A>
__device__ __forceinline__ void group_stage(typename A::T (&x)[1 << PS::K(R)], const Group<PS, R> &G,
                                            const typename A::W *stw, const A &ar)
{
    constexpr int K = PS::K(R), h = 1 << (K - 1 - k);
#pragma unroll
    for (int b = 0; b < (1 << k); ++b) {
        const typename A::W w = stw[G.tw(k, b)];
#pragma unroll
        for (int a = 0; a < h; ++a) {
            if (INV)
                ar.gs(x[b * 2 * h + a], x[b * 2 * h + a + h], w);
            else
                ar.ct(x[b * 2 * h + a], x[b * 2 * h + a + h], w);
        }
    }
}

template <class PS, int R, bool INV, class A>
__device__ __forceinline__ void group_stages(typename A::T (&x)[1 << PS::K(R)], const Group<PS, R> &G,
                                             const typename A::W *stw, const A &ar)
{
    constexpr int K = PS::K(R);
    if constexpr (!INV) {
        group_stage<PS, R, 0, false>(x, G, stw, ar);
        if constexpr (K > 1) group_stage<PS, R, 1, false>(x, G, stw, ar);
        if constexpr (K > 2) group_stage<PS, R, 2, false>(x, G, stw, ar);
        if constexpr (K > 3) group_stage<PS, R, 3, false>(x, G, stw, ar);
    } else {
        if constexpr (K > 3) group_stage<PS, R, 3, true>(x, G, stw, ar);
        if constexpr (K > 2) group_stage<PS, R, 2, true>(x, G, stw, ar);
        if constexpr (K > 1) group_stage<PS, R, 1, true>(x, G, stw, ar);
        group_stage<PS, R, 0, true>(x, G, stw, ar);
    }
}

// One round: every group of this thread is loaded (ld(sub, pos)), then
// `between()` runs (once, on every thread), then the groups are transformed
// and stored (st(sub, pos, value)).
template <class PS, int R, bool INV, class A, class Ld, class Between, class St>
__device__ __forceinline__ void round(const typename A::W *stw, const A &ar, Ld ld, Between between, St st)
{
    using Gr = Group<PS, R>;
    constexpr int P = Gr::per_thread, E = 1 << Gr::K;
    typename A::T x[P][E];
#pragma unroll
    for (int gi = 0; gi < P; ++gi) {
        const uint32_t g = threadIdx.x + gi * PS::threads;
        if (Gr::groups % PS::threads == 0 || g < Gr::groups) {
            const Gr G(g);
#pragma unroll
            for (int i = 0; i < E; ++i) x[gi][i] = ld(G.sub, G.pos(i));
        }
    }
    between();
#pragma unroll
    for (int gi = 0; gi < P; ++gi) {
        const uint32_t g = threadIdx.x + gi * PS::threads;
        if (Gr::groups % PS::threads == 0 || g < Gr::groups) {
            const Gr G(g);
            group_stages<PS, R, INV>(x[gi], G, stw, ar);
#pragma unroll
            for (int i = 0; i < E; ++i) st(G.sub, G.pos(i), x[gi][i]);
        }
    }
}

// the rounds from R up to (excluding) REND, through shared memory
template <class PS, int R, int REND, bool INV, class A>
__device__ __forceinline__ void middle_rounds(typename A::T *sm, const typename A::W *stw, const A &ar)
{
    if constexpr (R != REND) {
        round<PS, R, INV>(
            stw, ar, [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; }, [] {},
            [&](uint32_t sub, uint32_t pos, typename A::T v) { sm[sub * PS::pitch + pos] = v; });
        __syncthreads();
        middle_rounds<PS, (INV ? R - 1 : R + 1), REND, INV>(sm, stw, ar);
    }
}

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem)
{
    const uint32_t sa = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sa), "l"(gmem) : "memory");
}

// Stage the pass's twiddles (cp.async; waited by wait_twiddles).  `tab` is
// the transform's table: entry k is psi^brv(k) (forward) or psi^-brv(k)
// (inverse), 16 bytes each.
//   high pass  the entry of local stage j for position pos is 2^j + (pos >>
//              (s - j)) for every sub-transform: entries [0, 2^s) are copied;
//   low pass   sub-transform `sub` is row first + sub of the poly and its
//              entry is ((R1 + first + sub) << j) + t, t < 2^j; stage j's
//              entries are stored from (subs << j) - subs, t-major
//              ([t][sub]), so that adjacent sub-transforms read adjacent words.
template <int LOGN, class PS, class W>
__device__ __forceinline__ void stage_twiddles(W *stw, const W *tab, uint32_t first)
{
    static_assert(sizeof(W) == 16, "twiddles are copied in 16-byte units");
    if constexpr (PS::high) {
        for (uint32_t e = threadIdx.x; e < (1u << PS::s); e += PS::threads) cp_async16(&stw[e], &tab[e]);
    } else {
        const uint32_t u = (1u << Shape<LOGN>::n1) + first;
#pragma unroll 1
        for (int j = 0; j < PS::s; ++j) {
            const uint32_t cnt = PS::subs << j, off = cnt - PS::subs;
            for (uint32_t e = threadIdx.x; e < cnt; e += PS::threads)
                cp_async16(&stw[off + ((e & ((1u << j) - 1)) << PS::lsubs) + (e >> j)], &tab[(u << j) + e]);
        }
    }
    asm volatile("cp.async.commit_group;\n" ::: "memory");
}

__device__ __forceinline__ void wait_twiddles()
{
    asm volatile("cp.async.wait_all;\n" ::: "memory");
    __syncthreads();
}

// A coalesced sweep over the tile's elements e (tile / threads per thread):
// every load first, then every store.
template <class PS, class T, class Ld, class St>
__device__ __forceinline__ void sweep(Ld ld, St st)
{
    constexpr int P = (PS::tile + (int)PS::threads - 1) / (int)PS::threads;
    T v[P];
#pragma unroll
    for (int i = 0; i < P; ++i) {
        const uint32_t e = threadIdx.x + i * PS::threads;
        if (PS::tile % PS::threads == 0 || e < PS::tile) v[i] = ld(e);
    }
#pragma unroll
    for (int i = 0; i < P; ++i) {
        const uint32_t e = threadIdx.x + i * PS::threads;
        if (PS::tile % PS::threads == 0 || e < PS::tile) st(e, v[i]);
    }
}

// shared memory of a pass: staged twiddles, then the tile
template <class PS, class A>
struct Smem {
    typename A::W *stw;
    typename A::T *sm;
    __device__ __forceinline__ explicit Smem(uint8_t *raw)
        : stw(reinterpret_cast<typename A::W *>(raw)), sm(reinterpret_cast<typename A::T *>(stw + PS::tw_entries))
    {
    }
};

// ---------------------------------------------------------------------------
// Pass drivers.  `first` is the tile's first column (high) or row (low);
// the callbacks address the tile by (sub, pos), or by the element index e of
// a coalesced sweep, in which poly index = first * R2 + e (low pass).
// ---------------------------------------------------------------------------

// forward high pass: the first round loads directly (gload), the last stores
// directly (gstore)
template <int LOGN, class A, class GLoad, class GStore>
__device__ __forceinline__ void fwd_high_pass(uint8_t *raw, const typename A::W *tab, uint32_t first, const A &ar,
                                              GLoad gload, GStore gstore)
{
    using PS = HighPass<LOGN>;
    Smem<PS, A> S(raw);
    typename A::T *sm = S.sm;
    stage_twiddles<LOGN, PS>(S.stw, tab, first);
    auto sload = [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; };
    auto sstore = [&](uint32_t sub, uint32_t pos, typename A::T v) { sm[sub * PS::pitch + pos] = v; };
    if constexpr (PS::nr == 1) {
        round<PS, 0, false>(S.stw, ar, gload, wait_twiddles, gstore);
    } else {
        round<PS, 0, false>(S.stw, ar, gload, wait_twiddles, sstore);
        __syncthreads();
        middle_rounds<PS, 1, PS::nr - 1, false>(sm, S.stw, ar);
        round<PS, PS::nr - 1, false>(S.stw, ar, sload, [] {}, gstore);
    }
}

// forward low pass: the first round (lo fastest) loads directly; the last
// round goes through shared memory to a coalesced sweep epi(e, value), every
// value read by then (`pre()` runs before the first round)
template <int LOGN, class A, class Pre, class GLoad, class Epi>
__device__ __forceinline__ void fwd_low_pass(uint8_t *raw, const typename A::W *tab, uint32_t first, const A &ar,
                                             Pre pre, GLoad gload, Epi epi)
{
    using PS = LowPass<LOGN>;
    Smem<PS, A> S(raw);
    typename A::T *sm = S.sm;
    stage_twiddles<LOGN, PS>(S.stw, tab, first);
    pre();
    auto sstore = [&](uint32_t sub, uint32_t pos, typename A::T v) { sm[sub * PS::pitch + pos] = v; };
    round<PS, 0, false>(S.stw, ar, gload, wait_twiddles, sstore);
    __syncthreads();
    middle_rounds<PS, 1, PS::nr, false>(sm, S.stw, ar);
    epi([&](uint32_t e) { return sm[(e >> PS::s) * PS::pitch + (e & ((1u << PS::s) - 1))]; });
}

// inverse low pass: a coalesced sweep in (sweep_load(e)), the rounds, the
// last round (lo fastest) stores directly
template <int LOGN, class A, class SLoad, class GStore>
__device__ __forceinline__ void inv_low_pass(uint8_t *raw, const typename A::W *tab, uint32_t first, const A &ar,
                                             SLoad sweep_load, GStore gstore)
{
    using PS = LowPass<LOGN>;
    Smem<PS, A> S(raw);
    typename A::T *sm = S.sm;
    stage_twiddles<LOGN, PS>(S.stw, tab, first);
    sweep<PS, typename A::T>(sweep_load, [&](uint32_t e, typename A::T v) {
        sm[(e >> PS::s) * PS::pitch + (e & ((1u << PS::s) - 1))] = v;
    });
    wait_twiddles();
    middle_rounds<PS, PS::nr - 1, 0, true>(sm, S.stw, ar);
    round<PS, 0, true>(
        S.stw, ar, [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; }, [] {}, gstore);
}

// inverse high pass: the first round (sub-transforms fastest) loads
// directly, the last stores directly
template <int LOGN, class A, class GLoad, class GStore>
__device__ __forceinline__ void inv_high_pass(uint8_t *raw, const typename A::W *tab, uint32_t first, const A &ar,
                                              GLoad gload, GStore gstore)
{
    using PS = HighPass<LOGN>;
    Smem<PS, A> S(raw);
    typename A::T *sm = S.sm;
    stage_twiddles<LOGN, PS>(S.stw, tab, first);
    auto sload = [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; };
    auto sstore = [&](uint32_t sub, uint32_t pos, typename A::T v) { sm[sub * PS::pitch + pos] = v; };
    if constexpr (PS::nr == 1) {
        round<PS, 0, true>(S.stw, ar, gload, wait_twiddles, gstore);
    } else {
        round<PS, PS::nr - 1, true>(S.stw, ar, gload, wait_twiddles, sstore);
        __syncthreads();
        middle_rounds<PS, PS::nr - 2, 0, true>(sm, S.stw, ar);
        round<PS, 0, true>(S.stw, ar, sload, [] {}, gstore);
    }
}

// Per-limb modular tables, in device memory (built on the host once per
// context; the tables follow the array of these).
struct NttLimb {
    const ulonglong2 *fwd;   // [N]: (psi^brv(k), Shoup companion)
    const ulonglong2 *inv;   // [N]: (psi^-brv(k), Shoup companion)
    const ulonglong2 *qinv;  // [L]: q_j^-1 mod q (Shoup) for j > this limb, else (0, 0)
    uint64_t q;
    uint64_t mu64;           // floor(2^64 / q)
    ulonglong2 ninv;         // N^-1 mod q (Shoup)
};

// host: log2 of a power of two
inline uint32_t log2u(uint32_t N)
{
    uint32_t n = 0;
    while ((1u << n) < N) ++n;
    return n;
}

// host: bit reversal of the low `bits` bits
inline uint32_t bit_reverse(uint32_t k, uint32_t bits)
{
    uint32_t r = 0;
    for (uint32_t b = 0; b < bits; ++b) r = (r << 1) | ((k >> b) & 1u);
    return r;
}

}  // namespace fiona_ntt
