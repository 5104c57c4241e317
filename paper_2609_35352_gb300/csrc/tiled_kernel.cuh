// tiled_kernel.cuh -- the tiled evaluation kernel of the hybrid linear layer
// (instantiated by kernel_tiled.cu; its variants with signed-sum programs in
// the offset form by kernel_tiled_off.cu, and those for CTAs of at most 12
// warps by kernel_tiled_w12.cu: translation units built in parallel).
//
// A persistent CTA walks (limb l, coefficient tile) pairs, T = 32*C
// coefficients per tile, all outputs per tile.  Shared memory holds the
// schedule (bulk-copied once, completion counted on an mbarrier), the
// source region(s) and the partial sums.
//  1. The (c0, c1) tile of every input is copied into a source region, so
//     each input residue leaves HBM once.  With one coefficient per lane one
//     thread issues one or two TMA tensor copies (the inputs seen as a 3-D
//     tensor: coefficient, limb, input poly; a box of T coefficients, one
//     limb and up to 256 polys lands exactly in the region's layout), their
//     completion counted on the region's mbarrier; with two, every thread
//     copies its share with 16-byte cp.async (measured: the main loop of
//     those kernels compiles to fewer instructions that way).  With two
//     source regions the next tile's copies run during this tile; otherwise
//     warp 0 prefetches the next tile's inputs into L2.  Narrow plans (every
//     q < 2^52) with two coefficients per lane rewrite the tiles in
//     radix-2^26 split form (rns.cuh); with one, the sources stay canonical
//     and a product splits the words it reads.
//  2. The materialised shared signed sums (Sec. 4.2 "Sharing Signed Sums")
//     are formed once per tile, level by level, into the same region.
//  3. Each warp runs its operation stream (tiled.h): per scale group a
//     signed sum over sources (their shared-memory offsets read from the
//     schedule, or packed 16-bit indices where the larger schedule does not
//     fit), formed before the batch its product opens,
//     then one product by gamma (Sec. 4.2 "Grouping Reconstruction
//     Operations"); per raw term a PMult-MAC of a
//     plaintext tile and a source.  Plaintext tiles go from HBM straight to
//     registers: each warp keeps the next P (16, 8 or 4) of its stream in
//     flight, across job and tile boundaries, in a register queue indexed at
//     compile time (the stream is processed in batches of that many
//     operations).  Signed sums are lazy; products accumulate lazily; the
//     signed and raw routes are added before the single final reduction
//     (Sec. 4.2 "Combining the Signed and Raw Routes").
//  4. Outputs split across warps add their reduced partial sums.
//  5. The next tile's inputs are prepared (with two regions: their copies,
//     started at the top of this tile, waited for and rewritten) before the
//     one barrier per tile that publishes them.
// The waits are bounded: thread 0's wait for the schedule copy (about two
// seconds), and each thread's wait for a region's TMA copies and for the
// tensor-core contraction (TiledArgs::wait_ns, measured on the global
// timer; a wait also ends once another thread of the CTA gave up).  One
// that gives up raises the context's error flag; the CTA then stops at its
// next barrier (thread 0 first waits, bounded again, for the copies and the
// contraction it issued, and the CTA frees its tensor memory).  The tile in
// progress is computed from whatever its region holds, and the tiles the
// CTA did not reach stay unwritten: outputs are undefined after a timeout.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <mutex>

#include "async.cuh"
#include "tc_signed.cuh"
#include "tiled.h"
#include "tile_math.cuh"

namespace {

using namespace tile;

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

// TMA tensor copy of the box at (x, y, z) of the 3-D tensor map `tm` into
// shared memory at `dst` (128-byte aligned), counted on `bar`.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *tm, uint32_t x, uint32_t y, uint32_t z,
                                            uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

// bound of thread 0's wait, when a CTA stops, for the copies and the
// contraction it issued
constexpr uint64_t kDrainNs = 20000000;

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

// Per-thread asynchronous 16-byte copy global -> shared, tracked with
// commit groups (both addresses 16-byte aligned).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

template <uint32_t N>
__device__ __forceinline__ void cp_async_wait()
{
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// L2 policy for plaintexts: each is read once, so they go first when L2
// needs room (the staged input tiles and the schedule stay).
__device__ __forceinline__ uint64_t evict_first_policy()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

// OFF: the schedule's signed-sum programs are in the offset form (tiled.h;
// TiledArgs::src_offsets), each source address one addition.  WB: the most
// warps a CTA of this variant runs (fewer warps leave each thread more
// registers: the variants with 12 warps and 8-deep plaintext queues).  KA
// (with KC): every raw term of the plan has a constant plaintext, so every
// operation after a batch's first is constant or padding (a SEG only opens
// a batch): only the first operation of a batch tells its kind at run time
template <int C, bool NARROW, uint32_t P, bool KC, bool TC = false, bool OFF = false, uint32_t WB = kTiledMaxWarps,
          bool KA = false>
__global__ void __launch_bounds__(WB * 32)
    tiled_kernel(const TiledArgs a, const __grid_constant__ CUtensorMap tm_in)
{
    static_assert(!TC || (C == 1 && NARROW), "tensor-core sums: one coefficient per lane, narrow moduli");
    static_assert(!(TC && OFF), "tensor-core sums: packed programs");
    static_assert(!KA || KC, "every raw plaintext constant: the constant-plaintext variant");
    using A = Arith<NARROW>;
    using Acc = typename A::Acc;
    static_assert(P % 4 == 0, "operation words are read four at a time");
    constexpr bool TMA = C == 1;  // input tiles by TMA tensor copies
    // narrow sources in shared memory: split form (rewritten once per tile)
    // with two coefficients per lane; canonical, split where a product reads
    // them, with one (measured: VGG 2.46 -> 2.36 ms, while the layers with
    // two coefficients per lane ran 4-5% slower that way)
    constexpr bool SPLIT = NARROW && C == 2;
    constexpr uint32_t T = 32 * C;
    constexpr uint32_t TB = T * 8;  // bytes of one poly's tile
    constexpr uint32_t PB = 2 * TB; // bytes of one source (c0, c1)
    constexpr uint32_t VB = C * 8;  // bytes of one lane's words in a tile
    extern __shared__ __align__(128) char sm[];
    __shared__ int s_abort;
    if (threadIdx.x == 0) s_abort = 0;
    __shared__ __align__(16) LimbConst s_limb[2];  // per source region
    __shared__ uint32_t s_tmem;                    // TC: the CTA's tensor memory
    const uint32_t n_warps = blockDim.x >> 5;
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t n_buf = a.double_buffer ? 2 : 1;
    const uint32_t src0 = a.sched_bytes;  // byte offsets in `sm`
    const uint32_t part_base = src0 + n_buf * a.src_bytes;
    const uint32_t slot_base = part_base + a.n_part * PB;  // warp slots: n_slots tile pairs per warp
    const uint32_t bar_off = slot_base + a.n_slots * PB;  // the schedule copy's mbarrier
    const uint32_t bar0 = smem_addr(sm) + bar_off;
    const uint32_t bar_stage = bar0 + 8;  // + 8 * region: the region's input copies have landed
    const uint32_t bar_tc = bar0 + 24;    // TC: the tile's contraction is complete
    const uint32_t total = a.n_limbs * a.tiles_per_limb;
    const uint32_t lane_off = lane * VB;
    const uint32_t *sw = reinterpret_cast<const uint32_t *>(sm);
    const uint32_t zero = a.zero;  // 0, unknown to the compiler (rns::mac26)
    constexpr bool offsets = OFF;  // signed-sum runs hold source byte offsets (tiled.h)

    // the schedule, once per CTA (TMA copies want the regions 128-byte
    // aligned: a misaligned base raises the error flag and copies nothing)
    if (TMA && threadIdx.x == 0 && (smem_addr(sm) & 127u)) {
        s_abort = 1;
        atomicOr(a.err, 1);
    }
    __syncthreads();
    if (s_abort) return;
    if (threadIdx.x == 0) {
        if (TMA) {
            mbar_init(bar_stage, 1);
            mbar_init(bar_stage + 8, 1);
        }
        mbar_init(bar0, 1);
        mbar_expect_tx(bar0, a.sched_bytes);
        for (uint32_t o = 0; o < a.sched_bytes; o += 32768)
            bulk_g2s(smem_addr(sm) + o, reinterpret_cast<const char *>(a.sched) + o,
                     min(32768u, a.sched_bytes - o), bar0);
        s_abort = mbar_wait(bar0, 0) ? 0 : 1;
        if (s_abort) atomicOr(a.err, 1);
    }
    __syncthreads();
    if (s_abort) return;
    mbar_wait(bar0, 0);  // completed: orders the copied schedule before this thread's reads
    // the zero tile of each source region (read by NOP operations); published
    // by the first tile's barrier
    for (uint32_t i = threadIdx.x; i < n_buf * (PB / 16); i += blockDim.x) {
        const uint32_t reg = i / (PB / 16), o = i % (PB / 16);
        *reinterpret_cast<ulonglong2 *>(sm + src0 + reg * a.src_bytes + a.src_bytes - PB + o * 16) =
            make_ulonglong2(0, 0);
    }
    // TC: the tensor memory (published by the first tile's barrier) and the
    // contraction's barrier
    if constexpr (TC) {
        if (warp == 0) tcs::tmem_alloc(smem_addr(&s_tmem), a.tc_cols);
        if (threadIdx.x == 0) mbar_init(bar_tc, 1);
        tcs::fence_before();
    }

    // ---- this warp's operation stream and its plaintext queue
    const uint32_t wt = a.o_warp + warp * kWarpTableWords;
    const uint32_t op0 = sw[wt] * 4, n_batches = sw[wt + 1] / P;
    const uint32_t seg0 = sw[wt + 2] * 4, tg0 = sw[wt + 3];
    const uint32_t slots = slot_base + sw[wt + 4] * PB + lane_off;  // this lane's words of its warp's slot 0
    const uint64_t pol = evict_first_policy();
    const uint32_t stride_bytes = a.pt_stride * 8;  // L * N * 8 < 2^32 (lowering)
    auto tile_ptl = [&](uint32_t t) -> const char * {
        if (t >= total || !a.has_pt) return nullptr;
        const uint32_t l = a.limb0 + t / a.tiles_per_limb, k0 = (t % a.tiles_per_limb) * T;
        return reinterpret_cast<const char *>(a.pt + (size_t)l * a.N + k0 + lane * C);
    };
    // operation words (read-only while the kernel runs: plain loads the
    // compiler may schedule early)
    auto op_word = [&](uint32_t off) -> uint32_t { return *reinterpret_cast<const uint32_t *>(sm + off); };
    // the first words of plaintext 0 in the limb of the tile whose words
    // for this lane start at `ptl` (read by CONST operations)
    auto tile_limb = [&](const char *ptl, uint32_t t) -> const char * {
        return ptl ? ptl - ((t % a.tiles_per_limb) * T + lane * C) * 8 : nullptr;
    };
    // the plaintext words of operation word `w` in the tile at `base`, or
    // for a CONST operation in the limb at `lbase` (with stride 0 and the
    // schedule's own address for both when there is no next tile: a
    // harmless valid load)
    // (`i`: the operation's position in its batch)
    auto fetch = [&](const char *base, const char *lbase, uint32_t stride, uint32_t w, uint32_t i) -> V<C> {
        const char *b = KC && ((KA && i > 0) || (w & kOpConst)) ? lbase : base;
        return ldg_stream<C>(reinterpret_cast<const uint64_t *>(b + (uint64_t)(w >> kOpPtShift) * stride), pol);
    };
    V<C> r[P];
    uint32_t tile = blockIdx.x;
    const char *cur_ptl = tile_ptl(tile);
    const char *cur_lb = tile_limb(cur_ptl, tile);
    if (n_batches && tile < total) {
        const char *b0 = cur_ptl ? cur_ptl : reinterpret_cast<const char *>(a.sched);
        const char *l0 = cur_ptl ? cur_lb : b0;
        const uint32_t s0 = cur_ptl ? stride_bytes : 0;
#pragma unroll
        for (uint32_t i = 0; i < P; ++i) r[i] = fetch(b0, l0, s0, op_word(op0 + 4 * i), i);
    }

    // start the copies of tile `t`'s inputs into region `reg`: thread 0's
    // TMA copies (the boxes cover the 2 n_in polys, the last one ending at
    // the last poly: an overlap is copied twice, the same words), or every
    // thread's 16-byte asynchronous copies (one commit group per tile)
    constexpr uint32_t kChunks = TB / 16;  // 16-byte words per source poly
    const uint32_t n_chunks = 2 * a.n_in * kChunks;
    auto stage = [&](uint32_t t, uint32_t reg) {
        const uint32_t l = a.limb0 + t / a.tiles_per_limb, k0 = (t % a.tiles_per_limb) * T;
        const uint32_t dst = smem_addr(sm) + src0 + reg * a.src_bytes;
        if constexpr (TMA) {
            if (threadIdx.x != 0) return;
            const uint32_t bar = bar_stage + 8 * reg;
            // (test only: the CTA's first copy expects 16 bytes that never come)
            const uint32_t extra = (a.test_flags & kTiledFlagExtraTx) && t == blockIdx.x ? 16 : 0;
            mbar_expect_tx(bar, a.n_boxes * a.box_rows * TB + extra);
            for (uint32_t j = 0; j < a.n_boxes; ++j) {
                const uint32_t z = min(j * a.box_rows, 2 * a.n_in - a.box_rows);
                tma_load_3d(dst + z * TB, &tm_in, k0, l, z, bar);
            }
        } else {
            const char *base = reinterpret_cast<const char *>(a.in + (size_t)l * a.N + k0);
            const size_t LN8 = (size_t)a.L * a.N * 8;
            for (uint32_t i = threadIdx.x; i < n_chunks; i += blockDim.x)
                cp_async16(dst + i * 16, base + (size_t)(i / kChunks) * LN8 + (i % kChunks) * 16);
            cp_async_commit();
        }
    };
    uint32_t stage_phase = 0;  // bit r: phase of region r's copy barrier
    uint32_t failed = 0;       // 1 + region + 2 * phase of a copy wait that gave up
    uint32_t tc_phase = 0;     // TC: phase of the contraction's barrier
    uint32_t tc_failed = 0;    // TC: 1 + phase of a contraction wait that gave up

    // the tile's inputs in region `reg`, once the copies have landed (with
    // cp.async each thread rewrites the words it copied); and the tile's
    // limb constants
    auto prepare = [&](uint32_t t, uint32_t reg) {
        if (threadIdx.x == 0) s_limb[reg] = a.limbs[a.limb0 + t / a.tiles_per_limb];
        if (!a.n_in) return;
        if constexpr (TMA) {
            if (!async::mbar_wait_bounded(bar_stage + 8 * reg, (stage_phase >> reg) & 1u, &s_abort, a.wait_ns)) {
                s_abort = 1;  // the CTA stops after the next barrier
                atomicOr(a.err, 1);
                failed = 1 + reg + 2 * ((stage_phase >> reg) & 1u);
            }
            stage_phase ^= 1u << reg;
        } else {
            cp_async_wait<0>();  // this thread's copies; the barrier after publishes everyone's
        }
        if (SPLIT) {
            for (uint32_t i = threadIdx.x; i < n_chunks; i += blockDim.x) {
                ulonglong2 *p = reinterpret_cast<ulonglong2 *>(sm + src0 + reg * a.src_bytes + i * 16);
                const ulonglong2 x = *p;
                *p = make_ulonglong2(A::operand(x.x), A::operand(x.y));
            }
        }
    };

    // At the top of each tile its inputs and limb constants are in region
    // `buf`, published by a barrier.  With two regions the next tile's
    // copies are started at the top of this tile and prepared at its end,
    // where warps that finish early would otherwise wait: one barrier per
    // tile.  With one region the next tile is staged after every warp is
    // done with this one.
    uint32_t buf = 0;
    // after a copy wait gave up: every thread stops at the same barrier, once
    // thread 0 has waited (bounded again) for the copies it issued
    // (and for the tensor cores' work in flight), then frees the CTA's
    // tensor memory
    uint32_t tmem = 0;
    auto release = [&]() {
        if constexpr (TC) {
            tcs::fence_after();
            if (warp == 0) tcs::tmem_dealloc(tmem, a.tc_cols);
        }
    };
    auto stop = [&]() {
        const int never = 0;
        if (TMA && threadIdx.x == 0 && failed)
            async::mbar_wait_bounded(bar_stage + 8 * ((failed - 1) & 1), (failed - 1) >> 1, &never, kDrainNs);
        if (TC && threadIdx.x == 0 && tc_failed) async::mbar_wait_bounded(bar_tc, tc_failed - 1, &never, kDrainNs);
        if constexpr (TC) __syncthreads();
        release();
    };
    if (tile < total) {
        if (a.n_in) stage(tile, 0);
        prepare(tile, 0);
    }
    __syncthreads();
    if constexpr (TC) {
        tcs::fence_after();
        tmem = s_tmem;
    }
    if (s_abort) {
        stop();
        return;
    }
    for (; tile < total; tile += gridDim.x) {
        const uint32_t next = tile + gridDim.x;
        const char *next_ptl = tile_ptl(next);
        const char *next_lb = tile_limb(next_ptl, next);
        const uint32_t l = a.limb0 + tile / a.tiles_per_limb;
        const uint32_t k0 = (tile % a.tiles_per_limb) * T;
        const uint32_t lim = smem_addr(&s_limb[buf]);
        const uint32_t sb = src0 + buf * a.src_bytes;  // this tile's source region
        const uint32_t src = sb + lane_off;

        // 1. the next tile's inputs: into the other region, or (one region)
        //    into L2 ahead of their staging
        if (a.n_in && next < total) {
            if (a.double_buffer) {
                stage(next, buf ^ 1);
            } else if (warp == 0) {
                const uint32_t ln = a.limb0 + next / a.tiles_per_limb;
                const uint32_t kn = (next % a.tiles_per_limb) * T;
                for (uint32_t s = lane; s < 2 * a.n_in; s += 32)
                    prefetch_l2(a.in + ((size_t)s * a.L + ln) * a.N + kn, TB);
            }
        }

        // 2. TC: the scale groups' signed sums, as one contraction on the
        //    tensor cores (tc_signed.cuh): every warp converts its share of
        //    the inputs into tensor memory, one thread issues the
        //    contraction, and every warp turns its share of the products
        //    into canonical residues, stored as the group sources
        if constexpr (TC) {
            const TcGeometry geo{a.tc_k, a.tc_n};
            const uint32_t q4 = warp & 3, kq = warp >> 2, nq = n_warps >> 2;
            const uint32_t tq = tmem + ((32u * q4) << 16);
            const uint32_t row = sb + tcs::row_poly(q4) * TB + tcs::row_coef(q4, lane) * 8;
            tcs::convert(sm, row, PB, a.n_in, geo, tq, kq, nq);
            tcs::wait_st();
            tcs::fence_before();
            __syncthreads();
            tcs::fence_after();
            if (threadIdx.x == 0) tcs::issue(tmem, smem_addr(sm) + a.o_tcw * 4, geo, bar_tc);
            if (!async::mbar_wait_bounded(bar_tc, tc_phase, &s_abort, a.wait_ns)) {
                s_abort = 1;  // the CTA stops after this tile's last barrier
                atomicOr(a.err, 1);
                tc_failed = 1 + tc_phase;
            }
            tc_phase ^= 1;
            tcs::fence_after();
            const LimbConst m = load_limb(lim);
            const uint64_t bias = (uint64_t)a.tc_wabs * m.q;
            const float *magic = reinterpret_cast<const float *>(sm + a.o_tcm * 4);
            tcs::epilogue(tq, geo, a.tc_groups, magic, bias, m, lane, kq, nq, [&](uint32_t g, uint64_t v) {
                *reinterpret_cast<uint64_t *>(sm + row + (a.n_in + g) * PB) = v;
            });
            tcs::fence_before();
            __syncthreads();
        }
        // 2. materialised shared sums, children first (TC: its one level is
        //    the contraction)
        if constexpr (!TC)
        for (uint32_t lev = 0; lev < a.n_levels; ++lev) {
            for (uint32_t x = sw[a.o_level + lev] + warp; x < sw[a.o_level + lev + 1]; x += n_warps) {
                V<C> u0, u1;
                signed_sum<SPLIT, C, TB, NARROW && !SPLIT>(sm, src, sw[a.o_node_off + x] * 4, lim, 0, u0, u1, offsets);
                if constexpr (SPLIT) {  // stored in the sources' form
#pragma unroll
                    for (int x2 = 0; x2 < C; ++x2) {
                        u0.x[x2] = A::operand(u0.x[x2]);
                        u1.x[x2] = A::operand(u1.x[x2]);
                    }
                }
                const uint32_t dst = src + (a.n_in + x) * PB;
                sts<C>(sm, dst, u0);
                sts<C>(sm, dst + TB, u1);
            }
            __syncthreads();
        }

        // 3. this warp's operations, in batches of P; the plaintexts of the
        //    next batch are requested as these are consumed.  SEG and FOLD
        //    only open a batch and LAST only closes one, so the unrolled body
        //    has no branch: load, product-accumulate, request.
        Acc acc[2][C];
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int x = 0; x < C; ++x) A::zero(acc[c][x]);
        uint32_t sp = seg0, tp = tg0;
        // the job's result: reduce, store (output or partial slot), clear
        auto finish = [&]() {
            const LimbConst m = load_limb(lim);
            V<C> y0, y1;
#pragma unroll
            for (int x = 0; x < C; ++x) {
                y0.x[x] = A::reduce(acc[0][x], m);
                y1.x[x] = A::reduce(acc[1][x], m);
                A::zero(acc[0][x]);
                A::zero(acc[1][x]);
            }
            const uint32_t target = sw[tp++];
            if (target & kPartBit) {
                const uint32_t dst = part_base + (target & ~kPartBit) * PB + lane_off;
                sts<C>(sm, dst, y0);
                sts<C>(sm, dst + TB, y1);
            } else {
                uint64_t *dst = a.out + ((size_t)target * 2 * a.L + l) * a.N + k0 + lane * C;
                stg<C>(dst, y0);
                stg<C>(dst + (size_t)a.L * a.N, y1);
            }
        };
        for (uint32_t b = 0; b < n_batches; ++b) {
            const bool wrap = b + 1 == n_batches;
            const char *nb = wrap ? next_ptl : cur_ptl;
            const char *nlb = wrap ? next_lb : cur_lb;
            uint32_t ns = stride_bytes;
            if (!nb) {  // no next tile: a harmless valid load
                nb = nlb = reinterpret_cast<const char *>(a.sched);
                ns = 0;
            }
            const uint32_t cur_off = op0 + b * P * 4, next_off = wrap ? op0 : cur_off + P * 4;
            const uint32_t first = op_word(cur_off);
            if (first & kOpFold) {
                const LimbConst m = load_limb(lim);
#pragma unroll
                for (int c = 0; c < 2; ++c)
#pragma unroll
                    for (int x = 0; x < C; ++x) A::fold(acc[c][x], m);
            }
            V<C> g0, g1;  // the signed sum of this batch's SEG (operand form)
            const bool seg = first & kOpSeg;
            if (seg) {
                // shared signed sums this warp forms for its own later uses
                // (Sec. 4.2 "Sharing Signed Sums"), then this group's sum
                const uint32_t nf = first & (kOpMaxSources - 1);
                for (uint32_t f = 0; f < nf; ++f) {
                    // the target slot: the word before the program, or its
                    // third word in the offset form
                    const uint32_t dst = slots + sw[(sp >> 2) + (offsets ? 2 : 0)] * PB;
                    V<C> u0, u1;
                    sp = signed_sum<SPLIT, C, TB, NARROW && !SPLIT>(sm, src, offsets ? sp : sp + 4, lim, slots, u0, u1, offsets);
                    if constexpr (SPLIT) {  // stored in the sources' form
#pragma unroll
                        for (int x = 0; x < C; ++x) {
                            u0.x[x] = A::operand(u0.x[x]);
                            u1.x[x] = A::operand(u1.x[x]);
                        }
                    }
                    sts<C>(sm, dst, u0);
                    sts<C>(sm, dst + TB, u1);
                }
                sp = signed_sum<SPLIT, C, TB, NARROW && !SPLIT>(sm, src, sp, lim, slots, g0, g1, offsets);
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    g0.x[x] = A::operand(g0.x[x]);
                    g1.x[x] = A::operand(g1.x[x]);
                }
            }
            // this batch's and the next batch's operation words, four at a
            // time with 16-byte loads (every stream and batch starts on a
            // 16-byte boundary)
            uint4 cw4, nw4;
#pragma unroll
            for (uint32_t i = 0; i < P; ++i) {
                if (i % 4 == 0) {
                    cw4 = *reinterpret_cast<const uint4 *>(sm + cur_off + 4 * i);
                    nw4 = *reinterpret_cast<const uint4 *>(sm + next_off + 4 * i);
                }
                const uint32_t cwi = i % 4 == 0 ? cw4.x : i % 4 == 1 ? cw4.y : i % 4 == 2 ? cw4.z : cw4.w;
                const uint32_t nwi = i % 4 == 0 ? nw4.x : i % 4 == 1 ? nw4.y : i % 4 == 2 ? nw4.z : nw4.w;
                const uint32_t op = i == 0 ? first : cwi;
                V<C> s0, s1;
                if (i == 0 && seg) {
                    s0 = g0;
                    s1 = g1;
                } else {
                    const uint32_t so = src + (op & (kOpMaxSources - 1)) * PB;
                    s0 = lds<C>(sm, so);
                    s1 = lds<C>(sm, so + TB);
                    if constexpr (NARROW && !SPLIT) {  // canonical sources: the product's form here
#pragma unroll
                        for (int x = 0; x < C; ++x) {
                            s0.x[x] = A::operand(s0.x[x]);
                            s1.x[x] = A::operand(s1.x[x]);
                        }
                    }
                }
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    // a CONST plaintext is its limb's residue 0 at every coefficient
                    const bool cst = KC && x > 0 && ((KA && i > 0) || (op & kOpConst));
                    const uint64_t g = A::operand(cst ? r[i].x[0] : r[i].x[x]);
                    A::mac(acc[0][x], g, s0.x[x], zero);
                    A::mac(acc[1][x], g, s1.x[x], zero);
                }
                r[i] = fetch(nb, nlb, ns, nwi, i);
            }
            if (cw4.w & kOpLast) finish();  // the batch's last word
        }
        cur_ptl = next_ptl;
        cur_lb = next_lb;

        // 4. outputs split across warps: add the partial sums
        if (a.n_comb) {
            __syncthreads();
            const uint64_t q = load_limb(lim).q;
            for (uint32_t rr = warp; rr < a.n_comb; rr += n_warps) {
                V<C> y0{}, y1{};
                for (uint32_t pi = sw[a.o_comb_off + rr]; pi < sw[a.o_comb_off + rr + 1]; ++pi) {
                    const uint32_t ps = part_base + sw[a.o_comb_parts + pi] * PB + lane_off;
                    const V<C> v0 = lds<C>(sm, ps), v1 = lds<C>(sm, ps + TB);
#pragma unroll
                    for (int x = 0; x < C; ++x) {
                        y0.x[x] = rns::add_mod(y0.x[x], v0.x[x], q);
                        y1.x[x] = rns::add_mod(y1.x[x], v1.x[x], q);
                    }
                }
                uint64_t *dst = a.out + ((size_t)sw[a.o_comb_out + rr] * 2 * a.L + l) * a.N + k0 + lane * C;
                stg<C>(dst, y0);
                stg<C>(dst + (size_t)a.L * a.N, y1);
            }
        }
        // 5. the next tile: with two regions, prepare its inputs (their
        //    copies started at the top of this tile) before the barrier that
        //    publishes them; with one, stage them once every warp is done
        //    with this tile's region and partial slots.  The proxy fence
        //    orders this thread's shared-memory writes before the copies
        //    that will overwrite the region.
        if (a.double_buffer) {
            if (next < total) prepare(next, buf ^ 1);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncthreads();
            buf ^= 1;
        } else {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncthreads();
            if (next < total) {
                if (a.n_in) stage(next, 0);
                prepare(next, 0);
                __syncthreads();
            }
        }
        if (s_abort) {
            stop();
            return;
        }
    }
    release();
}

}  // namespace
