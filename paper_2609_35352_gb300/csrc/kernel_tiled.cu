// kernel_tiled.cu -- tiled evaluation of the hybrid linear layer.
//
// One CTA = one limb l and one tile of T = 32*C coefficients, all outputs.
//  1. Thread 0 copies the (c0, c1) tile of every input into shared memory
//     with bulk asynchronous copies (cp.async.bulk, completion counted on an
//     mbarrier): each input residue is read from HBM once per evaluation.
//     Narrow plans (every q < 2^52) then rewrite the tiles in radix-2^26
//     split form (rns.cuh), in place.
//  2. The shared signed sums U (Sec. 4.2 "Sharing Signed Sums") are formed
//     once per tile, level by level, into shared memory.
//  3. Each warp runs its jobs: per scale group a signed sum over shared
//     sources, then one product by gamma (Sec. 4.2 "Grouping Reconstruction
//     Operations"); per raw term a PMult-MAC with the plaintext streamed from
//     HBM (16-byte loads for C = 2) and the input read from shared memory.
//     A job first issues bulk L2 prefetches of all its plaintext tiles, so
//     the HBM latency overlaps its signed sums and earlier products.
//     Signed sums are lazy (plain 64-bit adds of + and - operands, folded
//     mod q only when a bound is reached); products accumulate lazily; the
//     signed and raw routes are added before the single final reduction
//     (Sec. 4.2 "Combining the Signed and Raw Routes").
//  4. Outputs split across warps add their reduced partial sums.
// The only wait is thread 0's bounded wait on the copy barrier; if it gives
// up, the CTA raises the context's error flag and leaves its tile unwritten.
#include <cuda_runtime.h>

#include "tiled.h"

namespace {

constexpr uint32_t kMaxThreads = kTiledMaxWarps * 32;
constexpr uint32_t kWaitLimit = 1u << 22;

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

// Bounded wait for phase `parity` of the barrier; false if it gave up.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    for (uint32_t it = 0; it < kWaitLimit; ++it) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(bar), "r"(parity)
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

// Any q < 2^60: 128-bit products (lo, hi), plain 64-bit signed sums.
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
    // a sum of at most `signed_budget` operands (each < q) stays below 2^64
    __device__ static uint64_t sum_value(uint64_t s, const LimbConst &m) { return rns::reduce64(s, m); }
};

// q < 2^52: split operands, three 64-bit product accumulators, packed sums.
template <>
struct Arith<true> {
    struct Acc {
        uint64_t lo, mid, hi;
    };
    __device__ static uint64_t operand(uint64_t a) { return rns::split26(a); }
    __device__ static void zero(Acc &a) { a.lo = a.mid = a.hi = 0; }
    __device__ static void mac(Acc &a, uint64_t x, uint64_t y) { rns::mac26(a.lo, a.mid, a.hi, x, y); }
    __device__ static uint64_t reduce(const Acc &a, const LimbConst &m)
    {
        return rns::reduce26(a.lo, a.mid, a.hi, m);
    }
    __device__ static void fold(Acc &a, const LimbConst &m)
    {
        a.lo = reduce(a, m);
        a.mid = a.hi = 0;
    }
    __device__ static uint64_t sum_value(uint64_t s, const LimbConst &m)
    {
        return rns::reduce64(rns::unsplit_sum(s), m);
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

template <int C>
__device__ __forceinline__ V<C> lds(const uint64_t *p)
{
    V<C> v;
    if constexpr (C == 2) {
        const ulonglong2 t = *reinterpret_cast<const ulonglong2 *>(p);
        v.x[0] = t.x;
        v.x[1] = t.y;
    } else {
        v.x[0] = *p;
    }
    return v;
}

template <int C>
__device__ __forceinline__ void st(uint64_t *p, const V<C> &v)
{
    if constexpr (C == 2) {
        *reinterpret_cast<ulonglong2 *>(p) = make_ulonglong2(v.x[0], v.x[1]);
    } else {
        *p = v.x[0];
    }
}

// Lazy signed sum of shared sources (both polys, C coefficients): plus- and
// minus-operands go into separate words, folded mod q when `budget`
// operands have gone in; returns the canonical sum in operand form.  The op
// list starts on a 16-byte boundary; op words are fetched four at a time,
// one group ahead of use.
template <bool NARROW, int C, uint32_t T>
__device__ __forceinline__ void signed_sum(const uint64_t *s_op, const uint32_t *ops, uint32_t b,
                                           uint32_t e, uint32_t kl, uint32_t budget,
                                           const LimbConst &m, V<C> &out0, V<C> &out1)
{
    using A = Arith<NARROW>;
    uint64_t P[2][C], M[2][C];
#pragma unroll
    for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int x = 0; x < C; ++x) P[c][x] = M[c][x] = 0;
    uint32_t cnt = 0;
    const uint4 *oq = reinterpret_cast<const uint4 *>(ops + b);
    const uint32_t n = e - b;
    uint4 cur = __ldg(oq);
    for (uint32_t o = 0; o < n; o += 4) {
        const uint4 nxt = __ldg(oq + o / 4 + 1);
        const uint32_t words[4] = {cur.x, cur.y, cur.z, cur.w};
#pragma unroll
        for (uint32_t t = 0; t < 4; ++t) {
            if (o + t >= n) break;
            const uint32_t w = words[t];
            const uint64_t *src = s_op + (size_t)(w & ~kNegBit) * 2 * T + kl;
            const V<C> v0 = lds<C>(src), v1 = lds<C>(src + T);
            if (cnt == budget) {
#pragma unroll
                for (int c = 0; c < 2; ++c)
#pragma unroll
                    for (int x = 0; x < C; ++x) {
                        P[c][x] = A::operand(A::sum_value(P[c][x], m));
                        M[c][x] = A::operand(A::sum_value(M[c][x], m));
                    }
                cnt = 1;
            }
            ++cnt;
            if (w & kNegBit) {
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    M[0][x] += v0.x[x];
                    M[1][x] += v1.x[x];
                }
            } else {
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    P[0][x] += v0.x[x];
                    P[1][x] += v1.x[x];
                }
            }
        }
        cur = nxt;
    }
#pragma unroll
    for (int x = 0; x < C; ++x) {
        out0.x[x] = A::operand(rns::sub_mod(A::sum_value(P[0][x], m), A::sum_value(M[0][x], m), m.q));
        out1.x[x] = A::operand(rns::sub_mod(A::sum_value(P[1][x], m), A::sum_value(M[1][x], m), m.q));
    }
}

template <int C, bool NARROW>
__global__ void __launch_bounds__(kMaxThreads) tiled_kernel(const TiledArgs a)
{
    using A = Arith<NARROW>;
    using Acc = typename A::Acc;
    constexpr uint32_t T = 32 * C;
    extern __shared__ __align__(16) uint64_t smem[];
    __shared__ int s_abort;
    const uint32_t n_warps = blockDim.x >> 5;
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t l = a.limb0 + blockIdx.y;
    const uint32_t k0 = blockIdx.x * T;
    const uint32_t kl = lane * C;  // this lane's first coefficient in the tile
    const LimbConst m = a.limbs[l];
    const size_t LN = (size_t)a.L * a.N;
    const uint32_t n_src = a.n_in + a.n_nodes;
    const uint32_t sum_budget = NARROW ? rns::kNarrowSumBudget : a.signed_budget;
    const uint32_t mac_budget = NARROW ? rns::kNarrowMacBudget : a.mac_budget;
    uint64_t *s_op = smem;                             // [n_src][2][T]
    uint64_t *s_part = smem + (size_t)n_src * 2 * T;   // [n_part][2][T]
    uint64_t *s_bar = s_part + (size_t)a.n_part * 2 * T;

    // 1. stage the input tiles
    if (a.n_in) {
        const uint32_t bar = smem_addr(s_bar);
        if (threadIdx.x == 0) {
            mbar_init(bar, 1);
            mbar_expect_tx(bar, a.n_in * 2 * T * 8);
            for (uint32_t s = 0; s < 2 * a.n_in; ++s)
                bulk_g2s(smem_addr(s_op + (size_t)s * T), a.in + ((size_t)s * a.L + l) * a.N + k0,
                         T * 8, bar);
            s_abort = mbar_wait(bar, 0) ? 0 : 1;
            if (s_abort) atomicExch(a.err, 1);
        }
        __syncthreads();
        if (s_abort) return;
        // the phase has completed: this returns at once and orders the
        // bulk-copied tiles before this thread's reads
        mbar_wait(bar, 0);
        if (NARROW) {
            for (uint32_t i = threadIdx.x; i < a.n_in * 2 * T; i += blockDim.x)
                s_op[i] = A::operand(s_op[i]);
            __syncthreads();
        }
    }

    // 2. shared signed sums, children first
    for (uint32_t lev = 0; lev < a.n_levels; ++lev) {
        for (uint32_t x = a.node_level_off[lev] + warp; x < a.node_level_off[lev + 1]; x += n_warps) {
            const uint32_t nd = a.node_slots[x];
            V<C> u0, u1;
            signed_sum<NARROW, C, T>(s_op, a.node_ops, a.node_op_off[2 * nd], a.node_op_off[2 * nd + 1],
                                     kl, sum_budget, m, u0, u1);
            uint64_t *dst = s_op + (size_t)(a.n_in + nd) * 2 * T + kl;
            st<C>(dst, u0);
            st<C>(dst + T, u1);
        }
        __syncthreads();
    }

    // 3. jobs
    const uint64_t *pt_tile = a.pt + (size_t)l * a.N + k0;
    const uint64_t *ptl = pt_tile + kl;
    for (uint32_t jb = a.warp_job_off[warp]; jb < a.warp_job_off[warp + 1]; ++jb) {
        const TiledJob job = a.jobs[jb];
        // start every plaintext tile of this job on its way into L2 (one
        // bulk prefetch per tile, spread over the lanes): the signed sums
        // below run while they arrive, and the loads that follow hit L2
        for (uint32_t t = job.raw_begin + lane; t < job.raw_end; t += 32)
            prefetch_l2(pt_tile + (size_t)a.raws[t].x * LN, T * 8);
        for (uint32_t sgi = job.seg_begin + lane; sgi < job.seg_end; sgi += 32)
            prefetch_l2(pt_tile + (size_t)a.segs[sgi].scale_pt * LN, T * 8);
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
            const V<C> g = ldg<C>(ptl + (size_t)sg.scale_pt * LN);
            V<C> s0, s1;
            signed_sum<NARROW, C, T>(s_op, a.ops, sg.op_begin, sg.op_end, kl, sum_budget, m, s0, s1);
            if (nprod + 1 > mac_budget) fold();
#pragma unroll
            for (int x = 0; x < C; ++x) {
                const uint64_t gx = A::operand(g.x[x]);
                A::mac(acc[0][x], gx, s0.x[x]);
                A::mac(acc[1][x], gx, s1.x[x]);
            }
            ++nprod;
        }

        // raw terms: (plaintext, input) pairs fetched two per 16-byte load,
        // one chunk ahead, so a chunk's U plaintext loads issue back to back
        constexpr uint32_t U = 8;
        const uint4 *rq = reinterpret_cast<const uint4 *>(a.raws + job.raw_begin);
        const uint32_t n_raw = job.raw_end - job.raw_begin;
        uint4 cur[U / 2];
#pragma unroll
        for (uint32_t i = 0; i < U / 2; ++i) cur[i] = __ldg(rq + i);
        uint32_t r = 0;
        for (; r + U <= n_raw; r += U) {
            V<C> pv[U];
#pragma unroll
            for (uint32_t i = 0; i < U / 2; ++i) {
                pv[2 * i] = ldg<C>(ptl + (size_t)cur[i].x * LN);
                pv[2 * i + 1] = ldg<C>(ptl + (size_t)cur[i].z * LN);
            }
            uint4 nxt[U / 2];
#pragma unroll
            for (uint32_t i = 0; i < U / 2; ++i) nxt[i] = __ldg(rq + (r + U) / 2 + i);
            // at most mac_budget products may sit in the accumulator
            if (nprod + U > mac_budget) fold();
#pragma unroll
            for (uint32_t u = 0; u < U; ++u) {
                const uint32_t in = (u & 1) ? cur[u / 2].w : cur[u / 2].y;
                const uint64_t *src = s_op + (size_t)in * 2 * T + kl;
                const V<C> v0 = lds<C>(src), v1 = lds<C>(src + T);
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    const uint64_t px = A::operand(pv[u].x[x]);
                    A::mac(acc[0][x], px, v0.x[x]);
                    A::mac(acc[1][x], px, v1.x[x]);
                }
            }
            nprod += U;
#pragma unroll
            for (uint32_t i = 0; i < U / 2; ++i) cur[i] = nxt[i];
        }
        for (; r < n_raw; ++r) {
            const uint2 t = a.raws[job.raw_begin + r];
            const V<C> pv = ldg<C>(ptl + (size_t)t.x * LN);
            const uint64_t *src = s_op + (size_t)t.y * 2 * T + kl;
            const V<C> v0 = lds<C>(src), v1 = lds<C>(src + T);
            if (nprod + 1 > mac_budget) fold();
#pragma unroll
            for (int x = 0; x < C; ++x) {
                const uint64_t px = A::operand(pv.x[x]);
                A::mac(acc[0][x], px, v0.x[x]);
                A::mac(acc[1][x], px, v1.x[x]);
            }
            ++nprod;
        }

        V<C> y0, y1;
#pragma unroll
        for (int x = 0; x < C; ++x) {
            y0.x[x] = A::reduce(acc[0][x], m);
            y1.x[x] = A::reduce(acc[1][x], m);
        }
        if (job.target & kPartBit) {
            uint64_t *dst = s_part + (size_t)(job.target & ~kPartBit) * 2 * T + kl;
            st<C>(dst, y0);
            st<C>(dst + T, y1);
        } else {
            uint64_t *dst = a.out + ((size_t)job.target * 2 * a.L + l) * a.N + k0 + kl;
            st<C>(dst, y0);
            st<C>(dst + LN, y1);
        }
    }

    // 4. outputs split across warps: add the partial sums
    if (a.n_comb) {
        __syncthreads();
        for (uint32_t r = warp; r < a.n_comb; r += n_warps) {
            V<C> y0{}, y1{};
            for (uint32_t q = a.comb_off[r]; q < a.comb_off[r + 1]; ++q) {
                const uint64_t *src = s_part + (size_t)a.comb_parts[q] * 2 * T + kl;
                const V<C> v0 = lds<C>(src), v1 = lds<C>(src + T);
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    y0.x[x] = rns::add_mod(y0.x[x], v0.x[x], m.q);
                    y1.x[x] = rns::add_mod(y1.x[x], v1.x[x], m.q);
                }
            }
            uint64_t *dst = a.out + ((size_t)a.comb_out[r] * 2 * a.L + l) * a.N + k0 + kl;
            st<C>(dst, y0);
            st<C>(dst + LN, y1);
        }
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
    dim3 grid(p->ctx->N / ts->tile, l1 - l0, 1);
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
