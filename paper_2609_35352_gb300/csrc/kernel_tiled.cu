// kernel_tiled.cu -- tiled evaluation of the hybrid linear layer.
//
// A persistent CTA walks (limb l, coefficient tile) pairs, T = 32*C
// coefficients per tile, all outputs per tile.  Shared memory holds the
// schedule (copied once), the source region(s), partial sums, and one
// plaintext ring per warp.
//  1. Thread 0 copies the (c0, c1) tile of every input into a source region
//     with bulk asynchronous copies (cp.async.bulk, completion counted on an
//     mbarrier), so each input residue leaves HBM once.  With two source
//     regions the next tile's copies run during this tile; otherwise warp 0
//     prefetches the next tile's inputs into L2.  Narrow plans (every
//     q < 2^52) rewrite the tiles in radix-2^26 split form (rns.cuh).
//  2. The shared signed sums U (Sec. 4.2 "Sharing Signed Sums") are formed
//     once per tile, level by level, into the same region.
//  3. Each warp runs its program: per scale group a signed sum over sources,
//     then one product by gamma (Sec. 4.2 "Grouping Reconstruction
//     Operations"); per raw term a PMult-MAC of a plaintext tile and a
//     source.  Plaintext tiles arrive through the warp's ring: each lane
//     copies its own C words of each tile D fetches ahead (cp.async, tracked
//     per thread with commit/wait groups), across job and tile boundaries,
//     and reads back only what it copied.  Signed sums are lazy; products
//     accumulate lazily; the signed and raw routes are added before the
//     single final reduction (Sec. 4.2 "Combining the Signed and Raw Routes").
//  4. Outputs split across warps add their reduced partial sums.
// The only spin-waits are thread 0's bounded mbarrier waits; if one gives up,
// the CTA raises the context's error flag, drains its own copies (bounded),
// and stops.
#include <cuda_runtime.h>

#include <algorithm>

#include "tiled.h"

namespace {

constexpr uint32_t kMaxThreads = kTiledMaxWarps * 32;
constexpr uint32_t kWaitLimit = 2000;
constexpr uint32_t kWaitHintNs = 1000000;

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// Bulk prefetch of `bytes` (a multiple of 16, 16-byte aligned) into L2.
__device__ __forceinline__ void prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Bounded wait for phase `parity` of the barrier; false if it gave up.  Each
// try suspends the thread for up to kWaitHintNs, so the wait ends after at
// most kWaitLimit * kWaitHintNs (about two seconds).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    for (uint32_t it = 0; it < kWaitLimit; ++it) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(bar), "r"(parity), "n"(kWaitHintNs)
            : "memory");
        if (ok) return true;
    }
    return false;
}

// Per-thread asynchronous copy of one lane's C words into shared memory.
template <int C>
__device__ __forceinline__ void cp_async(uint32_t dst, const uint64_t *src)
{
    if constexpr (C == 2)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
    else
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

template <uint32_t N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// A zero that the compiler cannot see through, computed from `v`: adding it
// to an address makes the address wait for the load that produced `v`.
__device__ __forceinline__ uint32_t opaque_zero(uint64_t v)
{
    uint32_t z;
    asm volatile("and.b32 %0, %1, 0;" : "=r"(z) : "r"((uint32_t)v));
    return z;
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
    __device__ static void mac(Acc &a, uint64_t x, uint64_t y) { rns::mac(a.lo, a.hi, x, y); }
    __device__ static uint64_t reduce(const Acc &a, const LimbConst &m) { return rns::reduce128(a.lo, a.hi, m); }
    __device__ static void fold(Acc &a, const LimbConst &m)
    {
        a.lo = reduce(a, m);
        a.hi = 0;
    }
};

// q < 2^52: every factor in split form (sources in shared memory, the other
// factor split on the way in); Karatsuba products into three accumulators;
// packed sums.
template <>
struct Arith<true> {
    struct Acc {
        uint64_t lo, x, hi;
    };
    __device__ static uint64_t operand(uint64_t a) { return rns::split26(a); }
    __device__ static void zero(Acc &a) { a.lo = a.x = a.hi = 0; }
    // both factors in operand (split) form
    __device__ static void mac(Acc &a, uint64_t x, uint64_t y) { rns::mac26(a.lo, a.x, a.hi, x, y); }
    __device__ static uint64_t reduce(const Acc &a, const LimbConst &m) { return rns::reduce26(a.lo, a.x, a.hi, m); }
    __device__ static void fold(Acc &a, const LimbConst &m)
    {
        a.lo = reduce(a, m);
        a.x = a.lo;  // the middle term x - lo - hi stays 0
        a.hi = 0;
    }
};

template <int C>
struct V {
    uint64_t x[C];
};

// shared-memory access through 32-bit addresses
template <int C>
__device__ __forceinline__ V<C> lds(uint32_t addr)
{
    V<C> v;
    if constexpr (C == 2)
        asm volatile("ld.shared.v2.u64 {%0, %1}, [%2];" : "=l"(v.x[0]), "=l"(v.x[1]) : "r"(addr));
    else
        asm volatile("ld.shared.u64 %0, [%1];" : "=l"(v.x[0]) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint32_t lds_u32(uint32_t addr)
{
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}

template <int C>
__device__ __forceinline__ void sts(uint32_t addr, const V<C> &v)
{
    if constexpr (C == 2)
        asm volatile("st.shared.v2.u64 [%0], {%1, %2};" ::"r"(addr), "l"(v.x[0]), "l"(v.x[1]) : "memory");
    else
        asm volatile("st.shared.u64 [%0], %1;" ::"r"(addr), "l"(v.x[0]) : "memory");
}

template <int C>
__device__ __forceinline__ void stg(uint64_t *p, const V<C> &v)
{
    if constexpr (C == 2)
        *reinterpret_cast<ulonglong2 *>(p) = make_ulonglong2(v.x[0], v.x[1]);
    else
        *p = v.x[0];
}

// Sum of n source tiles (both polys) whose words start at shared address
// `words`; `src` = this lane's address in the source region.
template <int C, uint32_t TB>
__device__ __forceinline__ void run_sum(uint32_t src, uint32_t words, uint32_t n, V<C> &s0, V<C> &s1)
{
    uint32_t k = 0;
    for (; k + 2 <= n; k += 2) {
        const uint32_t o0 = lds_u32(words + 4 * k), o1 = lds_u32(words + 4 * k + 4);
        const V<C> a0 = lds<C>(src + o0), b0 = lds<C>(src + o1);
        const V<C> a1 = lds<C>(src + o0 + TB), b1 = lds<C>(src + o1 + TB);
#pragma unroll
        for (int x = 0; x < C; ++x) {
            s0.x[x] += a0.x[x] + b0.x[x];
            s1.x[x] += a1.x[x] + b1.x[x];
        }
    }
    if (k < n) {
        const uint32_t o0 = lds_u32(words + 4 * k);
        const V<C> a0 = lds<C>(src + o0), a1 = lds<C>(src + o0 + TB);
#pragma unroll
        for (int x = 0; x < C; ++x) {
            s0.x[x] += a0.x[x];
            s1.x[x] += a1.x[x];
        }
    }
}

// Signed sum of the segment whose header word is at `hdr` (n_plus | n_minus
// << 16, then the words), both polys, reduced once to the canonical residue
// (narrow: from P - M + 64q, below 2^59 since each packed sum is below
// 2^58).  Returns the shared address just past the segment.
template <bool NARROW, int C, uint32_t TB>
__device__ __forceinline__ uint32_t signed_sum(uint32_t src, uint32_t hdr, const LimbConst &m,
                                               V<C> &o0, V<C> &o1)
{
    const uint32_t h = lds_u32(hdr);
    const uint32_t np = h & 0xffffu, nm = h >> 16;
    V<C> p0{}, p1{}, m0{}, m1{};
    run_sum<C, TB>(src, hdr + 4, np, p0, p1);
    run_sum<C, TB>(src, hdr + 4 + 4 * np, nm, m0, m1);
#pragma unroll
    for (int x = 0; x < C; ++x) {
        if constexpr (NARROW) {
            const uint64_t k = (uint64_t)rns::kNarrowSumBudget * m.q;
            o0.x[x] = rns::reduce64(rns::unsplit_sum(p0.x[x]) + k - rns::unsplit_sum(m0.x[x]), m);
            o1.x[x] = rns::reduce64(rns::unsplit_sum(p1.x[x]) + k - rns::unsplit_sum(m1.x[x]), m);
        } else {
            o0.x[x] = rns::sub_mod(rns::reduce64(p0.x[x], m), rns::reduce64(m0.x[x], m), m.q);
            o1.x[x] = rns::sub_mod(rns::reduce64(p1.x[x], m), rns::reduce64(m1.x[x], m), m.q);
        }
    }
    return hdr + 4 * (1 + np + nm);
}

template <int C, bool NARROW, uint32_t D>
__global__ void __launch_bounds__(kMaxThreads) tiled_kernel(const TiledArgs a)
{
    using A = Arith<NARROW>;
    using Acc = typename A::Acc;
    constexpr uint32_t T = 32 * C;
    constexpr uint32_t TB = T * 8;  // bytes of one poly's tile
    constexpr uint32_t VB = C * 8;  // bytes of one lane's words in a tile
    extern __shared__ __align__(16) uint64_t smem[];
    __shared__ int s_abort;
    const uint32_t n_warps = blockDim.x >> 5;
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t sch = smem_addr(smem);  // schedule words
    const uint32_t n_buf = a.double_buffer ? 2 : 1;
    const uint32_t src0 = sch + a.sched_bytes;
    const uint32_t part_base = src0 + n_buf * a.src_bytes;
    const uint32_t ring_base = part_base + a.n_part * 2 * TB;
    const uint32_t bar0 = ring_base + n_warps * D * TB;  // regions 0, 1; schedule
    const uint32_t total = a.n_limbs * a.tiles_per_limb;
    const uint32_t lane_off = lane * VB;
    auto sw = [&](uint32_t k) -> uint32_t { return lds_u32(sch + 4 * k); };

    // the schedule, once per CTA
    if (threadIdx.x == 0) {
        mbar_init(bar0, 1);
        mbar_init(bar0 + 8, 1);
        mbar_init(bar0 + 16, 1);
        mbar_expect_tx(bar0 + 16, a.sched_bytes);
        for (uint32_t o = 0; o < a.sched_bytes; o += 32768)
            bulk_g2s(sch + o, reinterpret_cast<const char *>(a.sched) + o, min(32768u, a.sched_bytes - o),
                     bar0 + 16);
        s_abort = mbar_wait(bar0 + 16, 0) ? 0 : 1;
        if (s_abort) atomicExch(a.err, 1);
    }
    __syncthreads();
    if (s_abort) return;
    mbar_wait(bar0 + 16, 0);

    // ---- this warp's plaintext ring
    const uint32_t f_begin = sw(a.o_fetch_off + warp);
    const uint32_t F = sw(a.o_fetch_off + warp + 1) - f_begin;
    const uint32_t my_tiles = blockIdx.x < total ? (total - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
    const uint32_t total_f = F * my_tiles;
    const uint32_t ring = ring_base + warp * D * TB + lane_off;
    auto tile_ptl = [&](uint32_t t) -> const uint64_t * {
        const uint32_t l = a.limb0 + t / a.tiles_per_limb, k0 = (t % a.tiles_per_limb) * T;
        return a.pt + (size_t)l * a.N + k0 + lane * C;
    };
    uint32_t p_next = 0, p_k = 0, p_tile = blockIdx.x;
    const uint64_t *p_ptl = tile_ptl(p_tile);
    // fetch p_next into its slot (or commit an empty group past the end)
    auto issue = [&](uint32_t dep) {
        if (p_next < total_f) {
            const uint32_t w = sw(f_begin + p_k);
            cp_async<C>(ring + (p_next % D) * TB + dep, p_ptl + ((uint64_t)w << a.log2N));
            if (++p_k == F) {
                p_k = 0;
                p_tile += gridDim.x;
                if (p_tile < total) p_ptl = tile_ptl(p_tile);
            }
        }
        cp_async_commit();
        ++p_next;
    };
    for (uint32_t i = 0; i < D; ++i) issue(0);
    uint32_t c_next = 0;
    // the next plaintext words of this lane; its slot is refilled D ahead,
    // after the read has landed (the refill address depends on it)
    auto consume = [&]() -> V<C> {
        cp_async_wait<D - 1>();
        const V<C> v = lds<C>(ring + (c_next % D) * TB);
        ++c_next;
        issue(opaque_zero(v.x[0]));
        return v;
    };
    // the next two, with one wait
    auto consume2 = [&](V<C> &v0, V<C> &v1) {
        cp_async_wait<D - 2>();
        v0 = lds<C>(ring + (c_next % D) * TB);
        v1 = lds<C>(ring + ((c_next + 1) % D) * TB);
        c_next += 2;
        issue(opaque_zero(v0.x[0]));
        issue(opaque_zero(v1.x[0]));
    };

    // thread 0: start the copies of tile `t` into region `r`
    auto stage = [&](uint32_t t, uint32_t r) {
        const uint32_t l = a.limb0 + t / a.tiles_per_limb, k0 = (t % a.tiles_per_limb) * T;
        const uint32_t bar = bar0 + 8 * r;
        mbar_expect_tx(bar, a.n_in * 2 * TB);
        const uint32_t dst = src0 + r * a.src_bytes;
        for (uint32_t s = 0; s < 2 * a.n_in; ++s)
            bulk_g2s(dst + s * TB, a.in + ((size_t)s * a.L + l) * a.N + k0, TB, bar);
    };

    uint32_t phase0 = 0, phase1 = 0, buf = 0;
    uint32_t tile = blockIdx.x;
    if (a.n_in && threadIdx.x == 0 && tile < total) stage(tile, 0);
    for (; tile < total; tile += gridDim.x) {
        const uint32_t next = tile + gridDim.x;
        const uint32_t l = a.limb0 + tile / a.tiles_per_limb;
        const uint32_t k0 = (tile % a.tiles_per_limb) * T;
        const LimbConst m = a.limbs[l];
        const uint32_t sb = src0 + buf * a.src_bytes;  // this tile's source region
        const uint32_t src = sb + lane_off;

        // 1. inputs of this tile
        if (a.n_in) {
            if (threadIdx.x == 0) {
                if (a.double_buffer && next < total) stage(next, buf ^ 1);
                s_abort = mbar_wait(bar0 + 8 * buf, buf ? phase1 : phase0) ? 0 : 1;
                if (s_abort) {
                    atomicExch(a.err, 1);
                    if (a.double_buffer && next < total) mbar_wait(bar0 + 8 * (buf ^ 1), buf ? phase0 : phase1);
                }
            }
            __syncthreads();
            if (s_abort) {
                cp_async_wait_all();
                return;
            }
            // the phase has completed: this returns at once and orders the
            // bulk-copied tiles before this thread's reads
            mbar_wait(bar0 + 8 * buf, buf ? phase1 : phase0);
            if (buf) phase1 ^= 1; else phase0 ^= 1;
            if (!a.double_buffer && next < total && warp == 0) {
                const uint32_t ln = a.limb0 + next / a.tiles_per_limb;
                const uint32_t kn = (next % a.tiles_per_limb) * T;
                for (uint32_t s = lane; s < 2 * a.n_in; s += 32)
                    prefetch_l2(a.in + ((size_t)s * a.L + ln) * a.N + kn, TB);
            }
            if (NARROW) {
                for (uint32_t i = threadIdx.x; i < a.n_in * 2 * T; i += blockDim.x) {
                    const uint32_t ad = sb + i * 8;
                    sts<1>(ad, V<1>{{A::operand(lds<1>(ad).x[0])}});
                }
                __syncthreads();
            }
        }

        // 2. shared signed sums, children first
        for (uint32_t lev = 0; lev < a.n_levels; ++lev) {
            for (uint32_t x = sw(a.o_level + lev) + warp; x < sw(a.o_level + lev + 1); x += n_warps) {
                const uint32_t nd = sw(a.o_node_slot + x);
                V<C> u0, u1;
                signed_sum<NARROW, C, TB>(src, sch + 4 * sw(a.o_node_prog_off + nd), m, u0, u1);
#pragma unroll
                for (int x2 = 0; x2 < C; ++x2) {
                    u0.x[x2] = A::operand(u0.x[x2]);
                    u1.x[x2] = A::operand(u1.x[x2]);
                }
                const uint32_t dst = src + (a.n_in + nd) * 2 * TB;
                sts<C>(dst, u0);
                sts<C>(dst + TB, u1);
            }
            __syncthreads();
        }

        // 3. this warp's program
        uint32_t jp = sch + 4 * sw(a.o_prog_off + warp);
        const uint32_t jend = sch + 4 * sw(a.o_prog_off + warp + 1);
        while (jp < jend) {
            const uint32_t target = lds_u32(jp), hdr = lds_u32(jp + 4);
            jp += 8;
            const uint32_t n_seg = hdr & 0xffffu, n_raw = hdr >> 16;
            Acc acc[2][C];
#pragma unroll
            for (int c = 0; c < 2; ++c)
#pragma unroll
                for (int x = 0; x < C; ++x) A::zero(acc[c][x]);
            uint32_t nprod = 0;
            auto fold = [&]() {
#pragma unroll
                for (int c = 0; c < 2; ++c)
#pragma unroll
                    for (int x = 0; x < C; ++x) A::fold(acc[c][x], m);
                nprod = 1;
            };

            for (uint32_t sgi = 0; sgi < n_seg; ++sgi) {
                V<C> s0, s1;
                jp = signed_sum<NARROW, C, TB>(src, jp, m, s0, s1);
                const V<C> g = consume();
                if (nprod + 1 > a.mac_budget) fold();
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    const uint64_t gx = A::operand(g.x[x]);
                    A::mac(acc[0][x], gx, A::operand(s0.x[x]));
                    A::mac(acc[1][x], gx, A::operand(s1.x[x]));
                }
                ++nprod;
            }
            // at most mac_budget products may sit in an accumulator: jobs
            // within the bound (all but extreme ones) skip the per-term checks
            const bool check = nprod + n_raw > a.mac_budget;
            uint32_t r = 0;
            for (; r + 2 <= n_raw; r += 2) {
                const uint32_t off0 = lds_u32(jp + 4 * r), off1 = lds_u32(jp + 4 * r + 4);
                V<C> p0, p1;
                consume2(p0, p1);
                const V<C> v00 = lds<C>(src + off0), v01 = lds<C>(src + off0 + TB);
                const V<C> v10 = lds<C>(src + off1), v11 = lds<C>(src + off1 + TB);
                if (check && nprod + 2 > a.mac_budget) fold();
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    const uint64_t q0 = A::operand(p0.x[x]), q1 = A::operand(p1.x[x]);
                    A::mac(acc[0][x], v00.x[x], q0);
                    A::mac(acc[1][x], v01.x[x], q0);
                    A::mac(acc[0][x], v10.x[x], q1);
                    A::mac(acc[1][x], v11.x[x], q1);
                }
                nprod += 2;
            }
            if (r < n_raw) {
                const uint32_t off = lds_u32(jp + 4 * r);
                const V<C> pv = consume();
                const V<C> v0 = lds<C>(src + off), v1 = lds<C>(src + off + TB);
                if (check && nprod + 1 > a.mac_budget) fold();
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    const uint64_t q = A::operand(pv.x[x]);
                    A::mac(acc[0][x], v0.x[x], q);
                    A::mac(acc[1][x], v1.x[x], q);
                }
                ++nprod;
            }
            jp += 4 * n_raw;

            V<C> y0, y1;
#pragma unroll
            for (int x = 0; x < C; ++x) {
                y0.x[x] = A::reduce(acc[0][x], m);
                y1.x[x] = A::reduce(acc[1][x], m);
            }
            if (target & kPartBit) {
                const uint32_t dst = part_base + (target & ~kPartBit) * 2 * TB + lane_off;
                sts<C>(dst, y0);
                sts<C>(dst + TB, y1);
            } else {
                uint64_t *dst = a.out + ((size_t)target * 2 * a.L + l) * a.N + k0 + lane * C;
                stg<C>(dst, y0);
                stg<C>(dst + (size_t)a.L * a.N, y1);
            }
        }

        // 4. outputs split across warps: add the partial sums
        if (a.n_comb) {
            __syncthreads();
            for (uint32_t r = warp; r < a.n_comb; r += n_warps) {
                V<C> y0{}, y1{};
                for (uint32_t q = sw(a.o_comb_off + r); q < sw(a.o_comb_off + r + 1); ++q) {
                    const uint32_t ps = part_base + sw(a.o_comb_parts + q) * 2 * TB + lane_off;
                    const V<C> v0 = lds<C>(ps), v1 = lds<C>(ps + TB);
#pragma unroll
                    for (int x = 0; x < C; ++x) {
                        y0.x[x] = rns::add_mod(y0.x[x], v0.x[x], m.q);
                        y1.x[x] = rns::add_mod(y1.x[x], v1.x[x], m.q);
                    }
                }
                uint64_t *dst = a.out + ((size_t)sw(a.o_comb_out + r) * 2 * a.L + l) * a.N + k0 + lane * C;
                stg<C>(dst, y0);
                stg<C>(dst + (size_t)a.L * a.N, y1);
            }
        }
        // every warp is done with this tile's region and partial slots; the
        // proxy fence orders this thread's shared-memory writes before the
        // bulk copies that will overwrite the region
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (a.n_in && !a.double_buffer && next < total && threadIdx.x == 0) stage(next, 0);
        buf ^= a.double_buffer;
    }
    cp_async_wait_all();
}

template <int C, bool NARROW>
void *select_depth(uint32_t depth)
{
    return depth == 16 ? reinterpret_cast<void *>(&tiled_kernel<C, NARROW, 16>)
                       : reinterpret_cast<void *>(&tiled_kernel<C, NARROW, 8>);
}

void *select_ptr(int C, bool narrow, uint32_t depth)
{
    if (C == 2) return narrow ? select_depth<2, true>(depth) : select_depth<2, false>(depth);
    return narrow ? select_depth<1, true>(depth) : select_depth<1, false>(depth);
}

}  // namespace

int tiled_kernel_attributes(int C, bool narrow, uint32_t depth, cudaFuncAttributes *attr)
{
    cudaError_t e = cudaFuncGetAttributes(attr, select_ptr(C, narrow, depth));
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel attributes: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

int tiled_configure_kernel(int C, bool narrow, uint32_t depth, size_t smem)
{
    cudaError_t e = cudaFuncSetAttribute(select_ptr(C, narrow, depth),
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel attribute: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

int launch_tiled(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt,
                 uint64_t *out, uint32_t l0, uint32_t l1)
{
    const TiledSchedule *ts = p->tiled;
    if (!ts) return set_error(FIONA_ERR_ARG, "tiled kernel not available for this plan");
    if (l1 <= l0) return FIONA_OK;
    TiledArgs a = ts->args;
    a.in = in;
    a.pt = pt;
    a.out = out;
    a.limb0 = l0;
    a.n_limbs = l1 - l0;
    const uint32_t tiles = a.n_limbs * a.tiles_per_limb;
    const uint32_t resident = ts->ctas_per_sm * (uint32_t)std::max(p->ctx->sm_count, 1);
    dim3 grid(std::min(tiles, resident));
    dim3 block(ts->warps * 32);
    cudaStream_t s = (cudaStream_t)stream;
    void *fn = select_ptr(ts->C, ts->narrow, ts->depth);
    void *args[] = {&a};
    cudaError_t e = cudaLaunchKernel(fn, grid, block, args, ts->smem, s);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}
