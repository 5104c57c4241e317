// rescale.cu -- the rescale that follows the layer: every output poly is
// divided by the last prime of its level (Sec. 2.2 "Homomorphic Operations":
// a PMult raises the scale and a rescale restores it; Sec. 4.2 "Combining
// the Signed and Raw Routes": one rescale per output).  For a poly y with
// limbs y_0..y_{Lc-1} in NTT form:
//   r    = coefficients of y_{Lc-1}       (inverse NTT mod q_{Lc-1})
//   y'_l = (y_l - NTT_l(r mod q_l)) * q_{Lc-1}^{-1}  mod q_l,   l < Lc-1.
// NTT form: A[k] = a(psi^(2 brv(k) + 1)) mod q, psi the least primitive
// 2N-th root of unity mod q, brv reversing the log2(N) bits of k.
//
// Transform structure.  The radix-2 stages of an N = 2^n point transform
// (Cooley-Tukey forward: at the stage with m blocks, block i pairs elements
// at distance N / 2m with twiddle psi^brv(m + i); Gentleman-Sande inverse
// with psi^-brv(m + i), then N^-1) are split between two passes over memory
// (N = R1 * R2, R1 = 2^floor(n/2)):
//   high pass  the first log2(R1) stages: for a fixed low index, the R1
//              elements hi * R2 + lo form one sub-transform; a CTA takes
//              tile / R1 of them (adjacent columns, so accesses coalesce);
//   low pass   the other stages, inside blocks of R2 consecutive elements;
//              a CTA takes tile / R2 blocks.
// A pass runs its stages in rounds of up to 4: in a round each thread holds
// the 2^K elements of one group in registers, spaced by the round's smallest
// distance, and applies the round's K stages to them (a group needs 2^K - 1
// twiddles).  Rounds hand over through shared memory ([sub-transform]
// [position], one word of padding per row against bank conflicts); the first
// and last rounds of a pass read and write global memory directly wherever
// their access pattern coalesces.  The CTA's twiddles are copied to shared
// memory (cp.async) while its data loads are in flight.  The forward stages
// run high pass then low pass; the inverse stages low then high.  Kernels
// are instantiated per log2 N, so all index arithmetic is constant-folded.
//
// Arithmetic.  Residues are 64-bit words and every modulus is below 2^60.
// A product by a table constant w uses Shoup's precomputed w' = floor(w 2^64
// / q): r = x w - floor(x w' / 2^64) q lies in [0, 2q) for any 64-bit x.  The
// quotient is taken from three of the four 32-bit partial products of x w'
// (the low-by-low one and the carries below bit 64 are dropped), which
// underestimates it by at most 2, so r lies in [0, 4q).  Values are kept
// lazily between stages:
//   forward, general   in [0, 8q): x is brought below 4q before each
//                      butterfly (x + t, x - t + 4q with t in [0, 4q));
//   forward, q < 2^56  (and q_{Lc-1} < 4 q_l) no reduction at all: each stage
//                      adds less than 4q to the bound, so after at most 17
//                      stages values stay below 72q < 2^63;
//   inverse            in [0, 4q): x + y is brought below 4q, and
//                      x - y + 4q is only multiplied.
// A pass makes its values canonical where it writes its final result.
//
// The rescale is four launches on the caller's stream: the two inverse passes
// on the last limb of every poly (in place: it becomes the coefficients r),
// then the two forward passes of every other limb; the first reads r and
// reduces it mod q_l, the second applies the subtraction and the product by
// q_{Lc-1}^{-1}.  The whole last limb must be known before any limb can be
// finished, so the rescale cannot share a launch with the layer's kernels,
// whose CTAs each see one tile of coefficients.
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "fiona_internal.h"

namespace {

typedef unsigned __int128 u128;

constexpr int kLogTileMax = 12;  // at most 4096 elements per CTA
constexpr uint32_t kThreads = 256;
constexpr int kLogNMin = 10, kLogNMax = 17;  // the ring dimensions a context accepts

// per limb, in device memory (the tables follow the array of these)
struct NttLimb {
    const ulonglong2 *fwd;   // [N]: (psi^brv(k), Shoup companion)
    const ulonglong2 *inv;   // [N]: (psi^-brv(k), Shoup companion)
    const ulonglong2 *qinv;  // [L]: q_j^-1 mod q (Shoup) for j > this limb, else (0, 0)
    uint64_t q;
    uint64_t mu64;           // floor(2^64 / q)
    ulonglong2 ninv;         // N^-1 mod q (Shoup)
};

// x w mod q up to 3q: in [0, 4q) (see the file comment)
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

// x mod q for any 64-bit x: floor(x * mu64 / 2^64) is floor(x / q) or one less
__device__ __forceinline__ uint64_t reduce_any(uint64_t x, uint64_t q, uint64_t mu64)
{
    return csub(x - __umul64hi(x, mu64) * q, q);
}

// Cooley-Tukey butterfly (x + w y, x - w y); see the file comment for ranges
template <bool FAST>
__device__ __forceinline__ void ct_bfly(uint64_t &x, uint64_t &y, ulonglong2 w, uint64_t q)
{
    const uint64_t a = FAST ? x : csub(x, 4 * q);
    const uint64_t t = mul_shoup_lazy(y, w, q);  // [0, 4q)
    x = a + t;
    y = a + 4 * q - t;
}

// Gentleman-Sande butterfly on [0, 4q): (x + y, w (x - y))
__device__ __forceinline__ void gs_bfly(uint64_t &x, uint64_t &y, ulonglong2 w, uint64_t q)
{
    const uint64_t a = x, b = y;
    x = csub(a + b, 4 * q);
    y = mul_shoup_lazy(a + 4 * q - b, w, q);
}

// ---------------------------------------------------------------------------
// Compile-time geometry
// ---------------------------------------------------------------------------
template <int LOGN>
struct Shape {
    static constexpr int n1 = LOGN / 2;
    static constexpr int lt = LOGN < kLogTileMax ? LOGN : kLogTileMax;  // log2(tile)
    static constexpr int ltiles = LOGN - lt;                            // log2(tiles per transform)
};

// A pass over a tile: 2^LSUBS sub-transforms of 2^S positions, in rounds.
template <int S, int LSUBS, bool HIGH>
struct PassShape {
    static constexpr int s = S, lsubs = LSUBS, subs = 1 << LSUBS;
    static constexpr int tile = 1 << (S + LSUBS);
    static constexpr int pitch = (1 << S) + 1;
    static constexpr int nr = (S + 3) / 4;
    __host__ __device__ static constexpr int K(int r) { return S / nr + (r < S % nr ? 1 : 0); }
    __host__ __device__ static constexpr int J0(int r) { return r == 0 ? 0 : J0(r - 1) + K(r - 1); }
    static constexpr bool high = HIGH;
    // shared memory: the staged twiddles (2^s entries for the high pass, at
    // most one per tile element for the low pass), then the padded tile
    static constexpr int tw_entries = HIGH ? 1 << S : 1 << (S + LSUBS);
    static constexpr size_t smem_bytes = sizeof(ulonglong2) * tw_entries + sizeof(uint64_t) * subs * pitch;
};

template <int LOGN>
using HighPass = PassShape<Shape<LOGN>::n1, Shape<LOGN>::lt - Shape<LOGN>::n1, true>;
template <int LOGN>
using LowPass = PassShape<LOGN - Shape<LOGN>::n1, Shape<LOGN>::lt - (LOGN - Shape<LOGN>::n1), false>;

// Group g of round R: sub-transform `sub`, and the element positions
// (hi << (lD + K)) + (i << lD) + lo, i < 2^K.  High pass: sub-transforms
// fastest (adjacent columns); low pass: lo fastest (adjacent elements).
template <class PS, int R>
struct Group {
    static constexpr int K = PS::K(R), J0 = PS::J0(R), LD = PS::s - J0 - K;
    static constexpr int groups = PS::tile >> K;
    static constexpr int per_thread = (groups + (int)kThreads - 1) / (int)kThreads;
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

template <class PS, int R, int k, bool INV, bool FAST>
__device__ __forceinline__ void group_stage(uint64_t (&x)[1 << PS::K(R)], const Group<PS, R> &G,
                                            const ulonglong2 *stw, uint64_t q)
{
    constexpr int K = PS::K(R), h = 1 << (K - 1 - k);
#pragma unroll
    for (int b = 0; b < (1 << k); ++b) {
        const ulonglong2 w = stw[G.tw(k, b)];
#pragma unroll
        for (int a = 0; a < h; ++a) {
            if (INV)
                gs_bfly(x[b * 2 * h + a], x[b * 2 * h + a + h], w, q);
            else
                ct_bfly<FAST>(x[b * 2 * h + a], x[b * 2 * h + a + h], w, q);
        }
    }
}

template <class PS, int R, bool INV, bool FAST>
__device__ __forceinline__ void group_stages(uint64_t (&x)[1 << PS::K(R)], const Group<PS, R> &G,
                                             const ulonglong2 *stw, uint64_t q)
{
    constexpr int K = PS::K(R);
    if constexpr (!INV) {
        group_stage<PS, R, 0, false, FAST>(x, G, stw, q);
        if constexpr (K > 1) group_stage<PS, R, 1, false, FAST>(x, G, stw, q);
        if constexpr (K > 2) group_stage<PS, R, 2, false, FAST>(x, G, stw, q);
        if constexpr (K > 3) group_stage<PS, R, 3, false, FAST>(x, G, stw, q);
    } else {
        if constexpr (K > 3) group_stage<PS, R, 3, true, FAST>(x, G, stw, q);
        if constexpr (K > 2) group_stage<PS, R, 2, true, FAST>(x, G, stw, q);
        if constexpr (K > 1) group_stage<PS, R, 1, true, FAST>(x, G, stw, q);
        group_stage<PS, R, 0, true, FAST>(x, G, stw, q);
    }
}

// One round: every group of this thread is loaded (ld(sub, pos)), then
// `between()` runs (once, on every thread), then the groups are transformed
// and stored (st(sub, pos, value)).
template <class PS, int R, bool INV, bool FAST, class Ld, class Between, class St>
__device__ __forceinline__ void round(const ulonglong2 *stw, uint64_t q, Ld ld, Between between, St st)
{
    using Gr = Group<PS, R>;
    constexpr int P = Gr::per_thread, E = 1 << Gr::K;
    uint64_t x[P][E];
#pragma unroll
    for (int gi = 0; gi < P; ++gi) {
        const uint32_t g = threadIdx.x + gi * kThreads;
        if (Gr::groups % kThreads == 0 || g < Gr::groups) {
            const Gr G(g);
#pragma unroll
            for (int i = 0; i < E; ++i) x[gi][i] = ld(G.sub, G.pos(i));
        }
    }
    between();
#pragma unroll
    for (int gi = 0; gi < P; ++gi) {
        const uint32_t g = threadIdx.x + gi * kThreads;
        if (Gr::groups % kThreads == 0 || g < Gr::groups) {
            const Gr G(g);
            group_stages<PS, R, INV, FAST>(x[gi], G, stw, q);
#pragma unroll
            for (int i = 0; i < E; ++i) st(G.sub, G.pos(i), x[gi][i]);
        }
    }
}

// the rounds strictly between the first and the last, through shared memory
template <class PS, int R, int REND, bool INV, bool FAST>
__device__ __forceinline__ void middle_rounds(uint64_t *sm, const ulonglong2 *stw, uint64_t q)
{
    if constexpr (R != REND) {
        round<PS, R, INV, FAST>(
            stw, q, [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; }, [] {},
            [&](uint32_t sub, uint32_t pos, uint64_t v) { sm[sub * PS::pitch + pos] = v; });
        __syncthreads();
        middle_rounds<PS, (INV ? R - 1 : R + 1), REND, INV, FAST>(sm, stw, q);
    }
}

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem)
{
    const uint32_t sa = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sa), "l"(gmem) : "memory");
}

// Stage the pass's twiddles (cp.async; waited by wait_twiddles).
//   high pass  the entry of local stage j for position pos is 2^j + (pos >>
//              (s - j)) for every sub-transform: entries [0, 2^s) are copied;
//   low pass   sub-transform `sub` is poly row first + sub and its entry is
//              ((R1 + first + sub) << j) + t, t < 2^j; stage j's entries
//              are stored from (subs << j) - subs, t-major ([t][sub]), so
//              that adjacent sub-transforms read adjacent words.
template <int LOGN, class PS>
__device__ __forceinline__ void stage_twiddles(ulonglong2 *stw, const ulonglong2 *tab, uint32_t first)
{
    if constexpr (PS::high) {
        for (uint32_t e = threadIdx.x; e < (1u << PS::s); e += kThreads) cp_async16(&stw[e], &tab[e]);
    } else {
        const uint32_t u = (1u << Shape<LOGN>::n1) + first;
#pragma unroll 1
        for (int j = 0; j < PS::s; ++j) {
            const uint32_t cnt = PS::subs << j, off = cnt - PS::subs;
            for (uint32_t e = threadIdx.x; e < cnt; e += kThreads)
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

// A coalesced sweep over the tile's elements e (tile / kThreads per thread):
// every load first, then every store.
template <class PS, class Ld, class St>
__device__ __forceinline__ void sweep(Ld ld, St st)
{
    constexpr int P = (PS::tile + (int)kThreads - 1) / (int)kThreads;
    uint64_t v[P];
#pragma unroll
    for (int i = 0; i < P; ++i) {
        const uint32_t e = threadIdx.x + i * kThreads;
        if (PS::tile % kThreads == 0 || e < PS::tile) v[i] = ld(e);
    }
#pragma unroll
    for (int i = 0; i < P; ++i) {
        const uint32_t e = threadIdx.x + i * kThreads;
        if (PS::tile % kThreads == 0 || e < PS::tile) st(e, v[i]);
    }
}

#define FIONA_SMEM(PS)                                          \
    extern __shared__ __align__(16) uint8_t smem_raw[];         \
    ulonglong2 *stw = reinterpret_cast<ulonglong2 *>(smem_raw); \
    uint64_t *sm = reinterpret_cast<uint64_t *>(stw + PS::tw_entries)

struct Args {
    uint64_t *polys;   // [count][Lc][N]
    uint64_t *out;     // [count][Lc-1][N]
    const NttLimb *T;
    uint32_t Lc;
};

// ---------------------------------------------------------------------------
// The four launches.  blockIdx.x = transform * tiles + tile; the transforms
// are the polys (inverse passes) or poly * (Lc - 1) + limb (forward passes).
// ---------------------------------------------------------------------------

// inverse, low stages, on the last limb in place: coalesced sweep in (the
// first round's groups are runs of adjacent elements), rounds, the last
// round (lo fastest) stores directly
template <int LOGN>
__global__ void __launch_bounds__(kThreads, 2) k_inv_low(Args A)
{
    using SH = Shape<LOGN>;
    using PS = LowPass<LOGN>;
    FIONA_SMEM(PS);
    const uint32_t tile = blockIdx.x & ((1u << SH::ltiles) - 1), p = blockIdx.x >> SH::ltiles;
    const uint32_t first = tile << PS::lsubs;
    uint64_t *g = A.polys + ((size_t)p * A.Lc + (A.Lc - 1)) * (1u << LOGN) + ((size_t)first << PS::s);
    const NttLimb &Tl = A.T[A.Lc - 1];
    const uint64_t q = Tl.q;
    stage_twiddles<LOGN, PS>(stw, Tl.inv, first);
    sweep<PS>([&](uint32_t e) { return g[e]; },
              [&](uint32_t e, uint64_t v) { sm[(e >> PS::s) * PS::pitch + (e & ((1u << PS::s) - 1))] = v; });
    wait_twiddles();
    middle_rounds<PS, PS::nr - 1, 0, true, false>(sm, stw, q);
    round<PS, 0, true, false>(
        stw, q, [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; }, [] {},
        [&](uint32_t sub, uint32_t pos, uint64_t v) { g[(sub << PS::s) + pos] = v; });
}

// inverse, high stages: the first round (sub-transforms fastest) loads
// directly, the last stores r = N^-1 x, canonical
template <int LOGN>
__global__ void __launch_bounds__(kThreads, 3) k_inv_high(Args A)
{
    using SH = Shape<LOGN>;
    using PS = HighPass<LOGN>;
    constexpr uint32_t R2 = 1u << (LOGN - SH::n1);
    FIONA_SMEM(PS);
    const uint32_t tile = blockIdx.x & ((1u << SH::ltiles) - 1), p = blockIdx.x >> SH::ltiles;
    const uint32_t first = tile << PS::lsubs;
    uint64_t *g = A.polys + ((size_t)p * A.Lc + (A.Lc - 1)) * (1u << LOGN) + first;
    const NttLimb &Tl = A.T[A.Lc - 1];
    const uint64_t q = Tl.q;
    const ulonglong2 ninv = Tl.ninv;
    stage_twiddles<LOGN, PS>(stw, Tl.inv, first);
    auto gload = [&](uint32_t sub, uint32_t pos) { return g[(size_t)pos * R2 + sub]; };
    auto sload = [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; };
    auto sstore = [&](uint32_t sub, uint32_t pos, uint64_t v) { sm[sub * PS::pitch + pos] = v; };
    auto gstore = [&](uint32_t sub, uint32_t pos, uint64_t v) {
        g[(size_t)pos * R2 + sub] = canon4(mul_shoup_lazy(v, ninv, q), q);
    };
    if constexpr (PS::nr == 1) {
        round<PS, 0, true, false>(stw, q, gload, wait_twiddles, gstore);
    } else {
        round<PS, PS::nr - 1, true, false>(stw, q, gload, wait_twiddles, sstore);
        __syncthreads();
        middle_rounds<PS, PS::nr - 2, 0, true, false>(sm, stw, q);
        round<PS, 0, true, false>(stw, q, sload, [] {}, gstore);
    }
}

// forward, high stages: r (the last limb's coefficients), reduced mod q_l
// unless FAST, loaded directly by the first round; the last round stores
// directly into out
template <int LOGN, bool FAST>
__global__ void __launch_bounds__(kThreads, 3) k_fwd_high(Args A)
{
    using SH = Shape<LOGN>;
    using PS = HighPass<LOGN>;
    constexpr uint32_t R2 = 1u << (LOGN - SH::n1);
    FIONA_SMEM(PS);
    const uint32_t tile = blockIdx.x & ((1u << SH::ltiles) - 1), tr = blockIdx.x >> SH::ltiles;
    const uint32_t p = tr / (A.Lc - 1), l = tr % (A.Lc - 1);
    const uint32_t first = tile << PS::lsubs;
    const uint64_t *g = A.polys + ((size_t)p * A.Lc + (A.Lc - 1)) * (1u << LOGN) + first;
    uint64_t *o = A.out + (size_t)tr * (1u << LOGN) + first;
    const NttLimb &Tl = A.T[l];
    const uint64_t q = Tl.q, mu = Tl.mu64;
    stage_twiddles<LOGN, PS>(stw, Tl.fwd, first);
    auto gload = [&](uint32_t sub, uint32_t pos) {
        const uint64_t v = g[(size_t)pos * R2 + sub];
        return FAST ? v : reduce_any(v, q, mu);
    };
    auto sload = [&](uint32_t sub, uint32_t pos) { return sm[sub * PS::pitch + pos]; };
    auto sstore = [&](uint32_t sub, uint32_t pos, uint64_t v) { sm[sub * PS::pitch + pos] = v; };
    auto gstore = [&](uint32_t sub, uint32_t pos, uint64_t v) { o[(size_t)pos * R2 + sub] = v; };
    if constexpr (PS::nr == 1) {
        round<PS, 0, false, FAST>(stw, q, gload, wait_twiddles, gstore);
    } else {
        round<PS, 0, false, FAST>(stw, q, gload, wait_twiddles, sstore);
        __syncthreads();
        middle_rounds<PS, 1, PS::nr - 1, false, FAST>(sm, stw, q);
        round<PS, PS::nr - 1, false, FAST>(stw, q, sload, [] {}, gstore);
    }
}

// forward, low stages: the first round (lo fastest) loads directly; the last
// round goes through shared memory to a coalesced sweep that writes
// y' = (y_l - t) * q_{Lc-1}^-1
template <int LOGN, bool FAST>
__global__ void __launch_bounds__(kThreads, 2) k_fwd_low(Args A)
{
    using SH = Shape<LOGN>;
    using PS = LowPass<LOGN>;
    FIONA_SMEM(PS);
    const uint32_t tile = blockIdx.x & ((1u << SH::ltiles) - 1), tr = blockIdx.x >> SH::ltiles;
    const uint32_t p = tr / (A.Lc - 1), l = tr % (A.Lc - 1);
    const uint32_t first = tile << PS::lsubs;
    uint64_t *o = A.out + (size_t)tr * (1u << LOGN) + ((size_t)first << PS::s);
    const uint64_t *y = A.polys + ((size_t)p * A.Lc + l) * (1u << LOGN) + ((size_t)first << PS::s);
    const NttLimb &Tl = A.T[l];
    const uint64_t q = Tl.q;
    const ulonglong2 qi = Tl.qinv[A.Lc - 1];
    stage_twiddles<LOGN, PS>(stw, Tl.fwd, first);
    // y is read only by the epilogue: start bringing it into L2 now
    for (uint32_t e = threadIdx.x * 16; e < PS::tile; e += kThreads * 16)
        asm volatile("prefetch.global.L2 [%0];\n" ::"l"(y + e));
    auto sstore = [&](uint32_t sub, uint32_t pos, uint64_t v) { sm[sub * PS::pitch + pos] = v; };
    round<PS, 0, false, FAST>(
        stw, q, [&](uint32_t sub, uint32_t pos) { return o[(sub << PS::s) + pos]; }, wait_twiddles, sstore);
    __syncthreads();
    middle_rounds<PS, 1, PS::nr, false, FAST>(sm, stw, q);
    // transform values: below 72q (FAST) or 8q; M = 128q or 8q bounds them
    const uint64_t M = (FAST ? 128 : 8) * q;
    sweep<PS>([&](uint32_t e) { return y[e]; },
              [&](uint32_t e, uint64_t v) {
                  const uint64_t t = sm[(e >> PS::s) * PS::pitch + (e & ((1u << PS::s) - 1))];
                  o[e] = canon4(mul_shoup_lazy(v + M - t, qi, q), q);
              });
}

// ---------------------------------------------------------------------------
// Host: tables, built once per context on its first rescale
// ---------------------------------------------------------------------------
uint64_t mulm(uint64_t a, uint64_t b, uint64_t q) { return (uint64_t)((u128)a * b % q); }

uint64_t powm(uint64_t b, uint64_t e, uint64_t q)
{
    uint64_t r = 1 % q;
    b %= q;
    for (; e; e >>= 1) {
        if (e & 1) r = mulm(r, b, q);
        b = mulm(b, b, q);
    }
    return r;
}

ulonglong2 shoup(uint64_t w, uint64_t q) { return make_ulonglong2(w, (uint64_t)(((u128)w << 64) / q)); }

uint32_t bit_reverse(uint32_t k, uint32_t bits)
{
    uint32_t r = 0;
    for (uint32_t b = 0; b < bits; ++b) r = (r << 1) | ((k >> b) & 1u);
    return r;
}

// The least primitive 2N-th root of unity mod q, or 0.  For the first x whose
// c = x^((q-1)/2N) has c^N = -1, c is primitive and the primitive roots are
// its odd powers; the least of them is returned.
uint64_t least_root(uint64_t q, uint32_t N)
{
    const uint64_t M = 2ull * N;
    if ((q - 1) % M) return 0;
    uint64_t g = 0;
    for (uint64_t x = 2; x < 1000000 && x < q; ++x) {
        const uint64_t c = powm(x, (q - 1) / M, q);
        if (powm(c, N, q) == q - 1) {
            g = c;
            break;
        }
    }
    if (!g) return 0;
    const uint64_t g2 = mulm(g, g, q);
    uint64_t best = g, cur = g;
    for (uint32_t j = 1; j < N; ++j) {
        cur = mulm(cur, g2, q);
        best = std::min(best, cur);
    }
    return best;
}

std::mutex g_ntt_mu;

int ensure_tables(const fiona_ctx *ctx)
{
    std::lock_guard<std::mutex> lock(g_ntt_mu);
    if (ctx->d_ntt) return FIONA_OK;
    const uint32_t N = ctx->N, L = ctx->L;
    uint32_t n = 0;
    while ((1u << n) < N) ++n;
    const size_t head = ((sizeof(NttLimb) * L + 255) / 256) * 256;
    const size_t table = sizeof(ulonglong2) * N, qtab = sizeof(ulonglong2) * L;
    const size_t per_limb = 2 * table + ((qtab + 255) / 256) * 256;
    const size_t bytes = head + per_limb * L;
    std::vector<uint8_t> host(bytes, 0);
    std::vector<uint64_t> pw(N);
    void *dev = nullptr;
    cudaError_t e = cudaMalloc(&dev, bytes);
    if (e != cudaSuccess) return set_error(FIONA_ERR_NOMEM, "rescale tables: %s", cudaGetErrorString(e));
    for (uint32_t l = 0; l < L; ++l) {
        const uint64_t q = ctx->moduli[l];
        const uint64_t psi = least_root(q, N);
        if (!psi) {
            cudaFree(dev);
            return set_error(FIONA_ERR_MODULUS, "rescale: modulus %u has no primitive 2N-th root of unity", l);
        }
        const size_t off = head + per_limb * l;
        ulonglong2 *fwd = reinterpret_cast<ulonglong2 *>(host.data() + off);
        ulonglong2 *inv = reinterpret_cast<ulonglong2 *>(host.data() + off + table);
        ulonglong2 *qinv = reinterpret_cast<ulonglong2 *>(host.data() + off + 2 * table);
        // powers of psi, then of psi^-1, placed in bit-reversed order
        for (int dir = 0; dir < 2; ++dir) {
            const uint64_t base = dir == 0 ? psi : powm(psi, q - 2, q);
            pw[0] = 1;
            for (uint32_t i = 1; i < N; ++i) pw[i] = mulm(pw[i - 1], base, q);
            ulonglong2 *dst = dir == 0 ? fwd : inv;
            for (uint32_t k = 0; k < N; ++k) dst[k] = shoup(pw[bit_reverse(k, n)], q);
        }
        for (uint32_t j = l + 1; j < L; ++j) qinv[j] = shoup(powm(ctx->moduli[j] % q, q - 2, q), q);
        NttLimb &T = reinterpret_cast<NttLimb *>(host.data())[l];
        const uint8_t *dbase = static_cast<const uint8_t *>(dev) + off;
        T.fwd = reinterpret_cast<const ulonglong2 *>(dbase);
        T.inv = reinterpret_cast<const ulonglong2 *>(dbase + table);
        T.qinv = reinterpret_cast<const ulonglong2 *>(dbase + 2 * table);
        T.q = q;
        T.mu64 = ~(uint64_t)0 / q;
        T.ninv = shoup(powm(N % q, q - 2, q), q);
    }
    e = cudaMemcpy(dev, host.data(), bytes, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        cudaFree(dev);
        return set_error(FIONA_ERR_CUDA, "rescale tables: %s", cudaGetErrorString(e));
    }
    ctx->d_ntt = dev;
    return FIONA_OK;
}

}  // namespace

int launch_rescale(const fiona_ctx *ctx, void *stream, uint32_t Lc, uint64_t count, uint64_t *polys, uint64_t *out)
{
    const int rc = ensure_tables(ctx);
    if (rc) return rc;
    if (count == 0) return FIONA_OK;
    uint32_t n = 0;
    while ((1u << n) < ctx->N) ++n;
    if (n < (uint32_t)kLogNMin || n > (uint32_t)kLogNMax)
        return set_error(FIONA_ERR_ARG, "rescale: N = %u outside [2^%d, 2^%d]", ctx->N, kLogNMin, kLogNMax);
    // the reduction-free forward butterflies need q < 2^56 and r < 4 q_l
    bool fast = true;
    const uint64_t qlast = ctx->moduli[Lc - 1];
    for (uint32_t l = 0; l + 1 < Lc; ++l)
        if (ctx->moduli[l] >= (1ull << 56) || qlast >= 4 * ctx->moduli[l]) fast = false;
    const uint32_t lt = std::min<uint32_t>(n, kLogTileMax), ltiles = n - lt;
    const int ix = (int)n - kLogNMin;
    typedef void (*Kern)(Args);
    static const Kern inv_low[] = {k_inv_low<10>, k_inv_low<11>, k_inv_low<12>, k_inv_low<13>,
                                   k_inv_low<14>, k_inv_low<15>, k_inv_low<16>, k_inv_low<17>};
    static const Kern inv_high[] = {k_inv_high<10>, k_inv_high<11>, k_inv_high<12>, k_inv_high<13>,
                                    k_inv_high<14>, k_inv_high<15>, k_inv_high<16>, k_inv_high<17>};
    static const Kern fwd_high[2][8] = {
        {k_fwd_high<10, false>, k_fwd_high<11, false>, k_fwd_high<12, false>, k_fwd_high<13, false>,
         k_fwd_high<14, false>, k_fwd_high<15, false>, k_fwd_high<16, false>, k_fwd_high<17, false>},
        {k_fwd_high<10, true>, k_fwd_high<11, true>, k_fwd_high<12, true>, k_fwd_high<13, true>,
         k_fwd_high<14, true>, k_fwd_high<15, true>, k_fwd_high<16, true>, k_fwd_high<17, true>}};
    static const Kern fwd_low[2][8] = {
        {k_fwd_low<10, false>, k_fwd_low<11, false>, k_fwd_low<12, false>, k_fwd_low<13, false>,
         k_fwd_low<14, false>, k_fwd_low<15, false>, k_fwd_low<16, false>, k_fwd_low<17, false>},
        {k_fwd_low<10, true>, k_fwd_low<11, true>, k_fwd_low<12, true>, k_fwd_low<13, true>,
         k_fwd_low<14, true>, k_fwd_low<15, true>, k_fwd_low<16, true>, k_fwd_low<17, true>}};
    const Kern ks[4] = {inv_low[ix], inv_high[ix], fwd_high[fast][ix], fwd_low[fast][ix]};
    static const size_t low_smem[] = {LowPass<10>::smem_bytes, LowPass<11>::smem_bytes, LowPass<12>::smem_bytes,
                                      LowPass<13>::smem_bytes, LowPass<14>::smem_bytes, LowPass<15>::smem_bytes,
                                      LowPass<16>::smem_bytes, LowPass<17>::smem_bytes};
    static const size_t high_smem[] = {HighPass<10>::smem_bytes, HighPass<11>::smem_bytes, HighPass<12>::smem_bytes,
                                       HighPass<13>::smem_bytes, HighPass<14>::smem_bytes, HighPass<15>::smem_bytes,
                                       HighPass<16>::smem_bytes, HighPass<17>::smem_bytes};
    const size_t smem[4] = {low_smem[ix], high_smem[ix], high_smem[ix], low_smem[ix]};
    cudaError_t e = cudaSuccess;
    {
        // the dynamic shared memory limit, once per device and kernel
        static bool configured[FIONA_MAX_DEVICES][kLogNMax - kLogNMin + 1][2] = {};
        std::lock_guard<std::mutex> lock(g_ntt_mu);
        if (ctx->device < 0 || ctx->device >= FIONA_MAX_DEVICES)
            return set_error(FIONA_ERR_ARG, "rescale: device %d", ctx->device);
        if (!configured[ctx->device][ix][fast]) {
            for (int i = 0; i < 4 && e == cudaSuccess; ++i)
                e = cudaFuncSetAttribute((const void *)ks[i], cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem[i]);
            if (e != cudaSuccess)
                return set_error(FIONA_ERR_CUDA, "rescale: kernel attributes: %s", cudaGetErrorString(e));
            configured[ctx->device][ix][fast] = true;
        }
    }
    // grid.x < 2^31: transforms * tiles, in chunks of whole polys
    const uint64_t max_polys = ((1ull << 31) - 1) / ((uint64_t)(Lc - 1) << ltiles);
    const NttLimb *T = reinterpret_cast<const NttLimb *>(ctx->d_ntt);
    cudaStream_t s = (cudaStream_t)stream;
    for (uint64_t p0 = 0; p0 < count && e == cudaSuccess; p0 += max_polys) {
        const uint64_t np = std::min<uint64_t>(count - p0, max_polys);
        Args a;
        a.polys = polys + p0 * Lc * (uint64_t)ctx->N;
        a.out = out + p0 * (Lc - 1) * (uint64_t)ctx->N;
        a.T = T;
        a.Lc = Lc;
        const uint32_t inv_blocks = (uint32_t)(np << ltiles);
        const uint32_t fwd_blocks = (uint32_t)((np * (Lc - 1)) << ltiles);
        ks[0]<<<inv_blocks, kThreads, smem[0], s>>>(a);
        ks[1]<<<inv_blocks, kThreads, smem[1], s>>>(a);
        ks[2]<<<fwd_blocks, kThreads, smem[2], s>>>(a);
        ks[3]<<<fwd_blocks, kThreads, smem[3], s>>>(a);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "rescale launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

void free_rescale_tables(const fiona_ctx *ctx)
{
    if (ctx->d_ntt) cudaFree(ctx->d_ntt);
    ctx->d_ntt = nullptr;
}
