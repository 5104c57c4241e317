// kernel_tiled.cu -- tiled evaluation of the hybrid linear layer.
//
// A persistent CTA walks (limb l, coefficient tile) pairs, T = 32*C
// coefficients per tile, all outputs per tile:
//  1. Thread 0 copies the (c0, c1) tile of every input into a shared-memory
//     source region with bulk asynchronous copies (cp.async.bulk, completion
//     counted on an mbarrier), so each input residue leaves HBM once.  With
//     two source regions the next tile's copies run during this tile;
//     otherwise warp 0 prefetches the next tile's inputs into L2.  Narrow
//     plans (every q < 2^52) rewrite the tiles in radix-2^26 split form
//     (rns.cuh), in place.
//  2. The shared signed sums U (Sec. 4.2 "Sharing Signed Sums") are formed
//     once per tile, level by level, into the same region.
//  3. Each warp runs its jobs: per scale group a signed sum over sources,
//     then one product by gamma (Sec. 4.2 "Grouping Reconstruction
//     Operations"); per raw term a PMult-MAC with the plaintext streamed from
//     HBM and the input read from shared memory.  Signed sums are lazy (plain
//     64-bit adds of plus and minus runs, reduced once); products accumulate
//     lazily; the signed and raw routes are added before the single final
//     reduction (Sec. 4.2 "Combining the Signed and Raw Routes").
//  4. Outputs split across warps add their reduced partial sums.
// The only waits are thread 0's bounded waits on the copy barriers; if one
// gives up, the CTA raises the context's error flag, waits (bounded) for any
// copy it still has in flight, and stops.
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

// ---------------------------------------------------------------------------
// Arithmetic policies.  "Operand form" is how residues sit in shared memory
// and registers before a product: canonical for Wide, split for Narrow.
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

// q < 2^52: shared sources in split form, plaintexts and signed sums as
// plain words; four 64-bit product accumulators; packed sums.
template <>
struct Arith<true> {
    struct Acc {
        uint64_t a00, a10, a01, a11;
    };
    __device__ static uint64_t operand(uint64_t a) { return rns::split26(a); }
    __device__ static void zero(Acc &a) { a.a00 = a.a10 = a.a01 = a.a11 = 0; }
    // x: a source in operand (split) form; y: any word below 2^59
    __device__ static void mac(Acc &a, uint64_t x, uint64_t y) { rns::mac26(a.a00, a.a10, a.a01, a.a11, x, y); }
    __device__ static uint64_t reduce(const Acc &a, const LimbConst &m)
    {
        return rns::reduce26(a.a00, a.a10, a.a01, a.a11, m);
    }
    __device__ static void fold(Acc &a, const LimbConst &m)
    {
        a.a00 = reduce(a, m);
        a.a10 = a.a01 = a.a11 = 0;
    }
};

template <int C>
struct V {
    uint64_t x[C];
};

template <int C>
__device__ __forceinline__ V<C> ldg(const uint64_t *p)
{
    V<C> v;
    if constexpr (C == 2) {
        const ulonglong2 t = __ldg(reinterpret_cast<const ulonglong2 *>(p));
        v.x[0] = t.x;
        v.x[1] = t.y;
    } else {
        v.x[0] = __ldg(p);
    }
    return v;
}

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

constexpr uint32_t kFull = 0xffffffffu;

// Sum of one run of n source tiles (both polys): the run's op words are read
// lane-parallel, 32 per coalesced load, and broadcast with shuffles.
template <int C, uint32_t TB>
__device__ __forceinline__ void run_sum(uint32_t src, const uint32_t *words, uint32_t n, uint32_t lane,
                                        V<C> &s0, V<C> &s1)
{
    for (uint32_t b0 = 0; b0 < n; b0 += 32) {
        const uint32_t nb = min(32u, n - b0);
        const uint32_t w = lane < nb ? __ldg(words + b0 + lane) : 0u;
        uint32_t k = 0;
        for (; k + 2 <= nb; k += 2) {
            const uint32_t o0 = __shfl_sync(kFull, w, k), o1 = __shfl_sync(kFull, w, k + 1);
            const V<C> a0 = lds<C>(src + o0), b0v = lds<C>(src + o1);
            const V<C> a1 = lds<C>(src + o0 + TB), b1 = lds<C>(src + o1 + TB);
#pragma unroll
            for (int x = 0; x < C; ++x) {
                s0.x[x] += a0.x[x] + b0v.x[x];
                s1.x[x] += a1.x[x] + b1.x[x];
            }
        }
        if (k < nb) {
            const uint32_t o0 = __shfl_sync(kFull, w, k);
            const V<C> a0 = lds<C>(src + o0), a1 = lds<C>(src + o0 + TB);
#pragma unroll
            for (int x = 0; x < C; ++x) {
                s0.x[x] += a0.x[x];
                s1.x[x] += a1.x[x];
            }
        }
    }
}

// Signed sum of one segment (plus run minus minus run), both polys.
// Narrow: returns P - M + 64q, a word below 2^59 congruent to the sum (the
// packed sums are below 2^58 each), ready to multiply without a reduction.
// Wide: returns the canonical sum.
template <bool NARROW, int C, uint32_t TB>
__device__ __forceinline__ void signed_sum(uint32_t src, const uint32_t *ops, const TiledSeg &sg,
                                           uint32_t lane, const LimbConst &m, V<C> &o0, V<C> &o1)
{
    V<C> p0{}, p1{}, m0{}, m1{};
    run_sum<C, TB>(src, ops + sg.op_begin, sg.n_plus, lane, p0, p1);
    run_sum<C, TB>(src, ops + sg.op_begin + sg.n_plus, sg.n_minus, lane, m0, m1);
#pragma unroll
    for (int x = 0; x < C; ++x) {
        if constexpr (NARROW) {
            const uint64_t k = (uint64_t)rns::kNarrowSumBudget * m.q;
            o0.x[x] = rns::unsplit_sum(p0.x[x]) + k - rns::unsplit_sum(m0.x[x]);
            o1.x[x] = rns::unsplit_sum(p1.x[x]) + k - rns::unsplit_sum(m1.x[x]);
        } else {
            o0.x[x] = rns::sub_mod(rns::reduce64(p0.x[x], m), rns::reduce64(m0.x[x], m), m.q);
            o1.x[x] = rns::sub_mod(rns::reduce64(p1.x[x], m), rns::reduce64(m1.x[x], m), m.q);
        }
    }
}

template <int C, bool NARROW>
__global__ void __launch_bounds__(kMaxThreads) tiled_kernel(const TiledArgs a)
{
    using A = Arith<NARROW>;
    using Acc = typename A::Acc;
    constexpr uint32_t T = 32 * C;
    constexpr uint32_t TB = T * 8;  // bytes of one poly's tile
    constexpr uint32_t U = 8 / C;   // raw terms per chunk
    extern __shared__ __align__(16) uint64_t smem[];
    __shared__ int s_abort;
    const uint32_t n_warps = blockDim.x >> 5;
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t base = smem_addr(smem);
    const uint32_t n_buf = a.double_buffer ? 2 : 1;
    const uint32_t part_base = base + n_buf * a.src_bytes;
    const uint32_t bar0 = part_base + a.n_part * 2 * TB;  // one 8-byte mbarrier per region
    const uint32_t total = a.n_limbs * a.tiles_per_limb;
    const uint32_t lane_off = lane * C * 8;
    if (threadIdx.x == 0) {
        mbar_init(bar0, 1);
        mbar_init(bar0 + 8, 1);
    }
    __syncthreads();

    // thread 0: start the copies of tile `t` into region `r`
    auto issue = [&](uint32_t t, uint32_t r) {
        const uint32_t l = a.limb0 + t / a.tiles_per_limb, k0 = (t % a.tiles_per_limb) * T;
        const uint32_t bar = bar0 + 8 * r;
        mbar_expect_tx(bar, a.n_in * 2 * TB);
        const uint32_t dst = base + r * a.src_bytes;
        for (uint32_t s = 0; s < 2 * a.n_in; ++s)
            bulk_g2s(dst + s * TB, a.in + ((size_t)s * a.L + l) * a.N + k0, TB, bar);
    };

    uint32_t phase0 = 0, phase1 = 0, buf = 0;
    uint32_t tile = blockIdx.x;
    if (a.n_in && threadIdx.x == 0 && tile < total) issue(tile, 0);
    for (; tile < total; tile += gridDim.x) {
        const uint32_t next = tile + gridDim.x;
        const uint32_t l = a.limb0 + tile / a.tiles_per_limb;
        const uint32_t k0 = (tile % a.tiles_per_limb) * T;
        const LimbConst m = a.limbs[l];
        const uint32_t sb = base + buf * a.src_bytes;  // this tile's source region
        const uint32_t src = sb + lane_off;

        // 1. inputs of this tile
        if (a.n_in) {
            if (threadIdx.x == 0) {
                if (a.double_buffer && next < total) issue(next, buf ^ 1);
                const uint32_t ph = buf ? phase1 : phase0;
                s_abort = mbar_wait(bar0 + 8 * buf, ph) ? 0 : 1;
                if (s_abort) {
                    atomicExch(a.err, 1);
                    if (a.double_buffer && next < total) mbar_wait(bar0 + 8 * (buf ^ 1), buf ? phase0 : phase1);
                }
            }
            __syncthreads();
            if (s_abort) return;
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
            for (uint32_t x = a.node_level_off[lev] + warp; x < a.node_level_off[lev + 1]; x += n_warps) {
                const uint32_t nd = a.node_slots[x];
                V<C> u0, u1;
                signed_sum<NARROW, C, TB>(src, a.ops, a.node_segs[nd], lane, m, u0, u1);
                if constexpr (NARROW) {
#pragma unroll
                    for (int x = 0; x < C; ++x) {
                        u0.x[x] = A::operand(rns::reduce64(u0.x[x], m));
                        u1.x[x] = A::operand(rns::reduce64(u1.x[x], m));
                    }
                }
                const uint32_t dst = src + (a.n_in + nd) * 2 * TB;
                sts<C>(dst, u0);
                sts<C>(dst + TB, u1);
            }
            __syncthreads();
        }

        // 3. jobs
        const uint64_t *pt_tile = a.pt + (size_t)l * a.N + k0;
        const uint64_t *ptl = pt_tile + lane * C;
        for (uint32_t jb = a.warp_job_off[warp]; jb < a.warp_job_off[warp + 1]; ++jb) {
            const TiledJob job = a.jobs[jb];

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

            for (uint32_t sgi = job.seg_begin; sgi < job.seg_end; ++sgi) {
                const TiledSeg sg = a.segs[sgi];
                const V<C> g = ldg<C>(ptl + ((uint64_t)sg.gamma_ptl << a.log2N));
                V<C> s0, s1;
                signed_sum<NARROW, C, TB>(src, a.ops, sg, lane, m, s0, s1);
                if (nprod + 1 > a.mac_budget) fold();
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    // gamma (a residue) in operand form times the signed sum
                    const uint64_t gx = A::operand(g.x[x]);
                    A::mac(acc[0][x], gx, s0.x[x]);
                    A::mac(acc[1][x], gx, s1.x[x]);
                }
                ++nprod;
            }

            // raw terms, 32 per batch: lane i holds term i's (plaintext index
            // * L, input offset); chunks of U plaintext loads are double
            // buffered, so one chunk's loads are in flight while the previous
            // chunk is multiplied
            const uint32_t n_raw = job.raw_end - job.raw_begin;
            for (uint32_t b0 = 0; b0 < n_raw; b0 += 32) {
                const uint32_t nb = min(32u, n_raw - b0);
                const uint2 d = __ldg(a.raws + job.raw_begin + b0 + min(lane, nb - 1));
                if (nprod + nb > a.mac_budget) fold();
                nprod += nb;
                V<C> pa[U], pb[U];
                auto load = [&](V<C>(&pv)[U], uint32_t c) {
#pragma unroll
                    for (uint32_t u = 0; u < U; ++u) {
                        // lanes past the batch hold a copy of its last term, so
                        // these loads stay valid; their products are skipped
                        const uint32_t ptl_i = __shfl_sync(kFull, d.x, c * U + u);
                        pv[u] = ldg<C>(ptl + ((uint64_t)ptl_i << a.log2N));
                    }
                };
                auto mul = [&](const V<C>(&pv)[U], uint32_t c) {
#pragma unroll
                    for (uint32_t u = 0; u < U; ++u) {
                        const uint32_t i = c * U + u;
                        const uint32_t off = __shfl_sync(kFull, d.y, i);
                        if (i < nb) {
                            const V<C> v0 = lds<C>(src + off), v1 = lds<C>(src + off + TB);
#pragma unroll
                            for (int x = 0; x < C; ++x) {
                                A::mac(acc[0][x], v0.x[x], pv[u].x[x]);
                                A::mac(acc[1][x], v1.x[x], pv[u].x[x]);
                            }
                        }
                    }
                };
                const uint32_t n_chunks = (nb + U - 1) / U;
                load(pa, 0);
                for (uint32_t c = 0; c < n_chunks; c += 2) {
                    if (c + 1 < n_chunks) load(pb, c + 1);
                    mul(pa, c);
                    if (c + 1 < n_chunks) {
                        if (c + 2 < n_chunks) load(pa, c + 2);
                        mul(pb, c + 1);
                    }
                }
            }

            V<C> y0, y1;
#pragma unroll
            for (int x = 0; x < C; ++x) {
                y0.x[x] = A::reduce(acc[0][x], m);
                y1.x[x] = A::reduce(acc[1][x], m);
            }
            if (job.target & kPartBit) {
                const uint32_t dst = part_base + (job.target & ~kPartBit) * 2 * TB + lane_off;
                sts<C>(dst, y0);
                sts<C>(dst + TB, y1);
            } else {
                uint64_t *dst = a.out + ((size_t)job.target * 2 * a.L + l) * a.N + k0 + lane * C;
                stg<C>(dst, y0);
                stg<C>(dst + (size_t)a.L * a.N, y1);
            }
        }

        // 4. outputs split across warps: add the partial sums
        if (a.n_comb) {
            __syncthreads();
            for (uint32_t r = warp; r < a.n_comb; r += n_warps) {
                V<C> y0{}, y1{};
                for (uint32_t q = a.comb_off[r]; q < a.comb_off[r + 1]; ++q) {
                    const uint32_t ps = part_base + a.comb_parts[q] * 2 * TB + lane_off;
                    const V<C> v0 = lds<C>(ps), v1 = lds<C>(ps + TB);
#pragma unroll
                    for (int x = 0; x < C; ++x) {
                        y0.x[x] = rns::add_mod(y0.x[x], v0.x[x], m.q);
                        y1.x[x] = rns::add_mod(y1.x[x], v1.x[x], m.q);
                    }
                }
                uint64_t *dst = a.out + ((size_t)a.comb_out[r] * 2 * a.L + l) * a.N + k0 + lane * C;
                stg<C>(dst, y0);
                stg<C>(dst + (size_t)a.L * a.N, y1);
            }
        }
        // every warp is done with this tile's region and partial slots; the
        // proxy fence orders this thread's shared-memory writes before the
        // bulk copies that will overwrite the region
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (a.n_in && !a.double_buffer && next < total && threadIdx.x == 0) issue(next, 0);
        buf ^= a.double_buffer;
    }
}

void *select_ptr(int C, bool narrow)
{
    if (C == 2)
        return narrow ? reinterpret_cast<void *>(&tiled_kernel<2, true>)
                      : reinterpret_cast<void *>(&tiled_kernel<2, false>);
    return narrow ? reinterpret_cast<void *>(&tiled_kernel<1, true>)
                  : reinterpret_cast<void *>(&tiled_kernel<1, false>);
}

}  // namespace

int tiled_kernel_attributes(int C, bool narrow, cudaFuncAttributes *attr)
{
    cudaError_t e = cudaFuncGetAttributes(attr, select_ptr(C, narrow));
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel attributes: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

int tiled_configure_kernel(int C, bool narrow, size_t smem)
{
    cudaError_t e = cudaFuncSetAttribute(select_ptr(C, narrow),
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
    if (ts->C == 2) {
        if (ts->narrow)
            tiled_kernel<2, true><<<grid, block, ts->smem, s>>>(a);
        else
            tiled_kernel<2, false><<<grid, block, ts->smem, s>>>(a);
    } else {
        if (ts->narrow)
            tiled_kernel<1, true><<<grid, block, ts->smem, s>>>(a);
        else
            tiled_kernel<1, false><<<grid, block, ts->smem, s>>>(a);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "tiled kernel launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}
