// kernel_ws.cu -- warp-specialised tiled evaluation of the hybrid linear
// layer, two coefficients per lane (T = 64 coefficients per tile).
//
// Same work as kernel_tiled.cu (one persistent CTA per SM walks the (limb,
// coefficient tile) pairs; every input residue leaves HBM once; signed sums,
// scale products and raw PMult-MACs accumulate in registers; one reduction
// per output), with the input staging taken off the warps that compute:
//   * the stager warp copies each tile's (c0, c1) input tiles into a source
//     region by TMA tensor copies (boxes of 64 coefficients x 1 limb x up to
//     256 polys), waits for them and, for narrow plans (every q < 2^52),
//     rewrites them in radix-2^26 split form; then it publishes the region
//     on an mbarrier.  One or two regions: with two, the next tile's inputs
//     land while this tile is computed.  The consumer warps release a region
//     on another mbarrier.
//   * each consumer warp runs its operation stream in batches of P
//     operations (tiled.h).  Its plaintext tiles go from HBM into a ring of
//     D groups of P slots in shared memory by per-lane 16-byte asynchronous
//     copies, D - 1 batches ahead of their use, across tile boundaries (each
//     lane reads back only the words it copied, so no warp-level
//     synchronisation is needed); padding operations get no copy.  Per scale
//     group a signed sum (Sec. 4.2 "Grouping Reconstruction Operations") and
//     one product by gamma; per raw term a PMult-MAC; the signed and raw
//     routes are added before the single reduction (Sec. 4.2 "Combining the
//     Signed and Raw Routes").  Outputs split across warps add their reduced
//     partial sums after an mbarrier of the consumer warps.
// Every wait is bounded in time (WsArgs::wait_ns): a wait that gives up
// raises the context's error flag and makes every warp of the CTA stop; the
// stager then waits (bounded again) for the copies it issued to land before
// it exits.  The outputs are undefined after such a failure.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstring>

#include "async.cuh"
#include "tile_math.cuh"
#include "tiled.h"

namespace {

using namespace tile;
using namespace async;

constexpr int C = 2;
constexpr uint32_t T = 64;         // coefficients per tile
constexpr uint32_t TB = T * 8;     // bytes of one poly's tile
constexpr uint32_t PB = 2 * TB;    // bytes of one source (c0, c1)
constexpr uint32_t VB = C * 8;     // bytes of one lane's words in a tile
constexpr uint64_t kDrainNs = 20000000;  // bound of the stager's wait for its copies when a CTA stops

// MAXW: most consumer warps of a launch.  Sixteen consumer warps and the two
// data-movement warps allow 96 registers a thread; fourteen allow 128.
template <bool NARROW, uint32_t P, bool KC, uint32_t MAXW, uint32_t D>
__global__ void __launch_bounds__((MAXW + 1) * 32, 1)
    ws_kernel(const WsArgs a, const __grid_constant__ CUtensorMap tm_in)
{
    using A = Arith<NARROW>;
    using Acc = typename A::Acc;
    static_assert(P == 4, "operation words are read four at a time");
    static_assert(D >= 2, "the ring holds the batch in use and the ones in flight");
    constexpr bool SPLIT = NARROW;  // sources in split form in shared memory
    extern __shared__ __align__(128) char sm[];
    __shared__ int s_abort;
    __shared__ __align__(16) LimbConst s_limb[2];
    const uint32_t W = (blockDim.x >> 5) - 1;  // consumer warps
    const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const WsLayout lay(a.smem_sched_bytes, a.n_buf, a.src_bytes, a.n_part, W, D, P, TB, a.n_slots);
    const uint32_t smb = smem_addr(sm);
    const uint32_t bar_sched = smb + lay.bar0;
    auto bar_loaded = [&](uint32_t r) { return bar_sched + 8 + 8 * r; };
    auto bar_ready = [&](uint32_t r) { return bar_sched + 24 + 8 * r; };
    auto bar_rempty = [&](uint32_t r) { return bar_sched + 40 + 8 * r; };
    const uint32_t bar_comb = bar_sched + 56;  // consumers' barrier before combining partial sums
    const uint32_t total = a.n_limbs * a.tiles_per_limb;
    const uint32_t *sw = reinterpret_cast<const uint32_t *>(sm);
    volatile int *abort_flag = &s_abort;
    auto fail = [&]() {
        *abort_flag = 1;
        atomicOr(a.err, 1);
    };

    if (threadIdx.x == 0) {
        s_abort = 0;
        if (smb & 127u) {  // TMA destinations want 128-byte alignment
            s_abort = 1;
            atomicOr(a.err, 1);
        } else {
            mbar_init(bar_sched, 1);
            for (uint32_t r = 0; r < 2; ++r) {
                mbar_init(bar_loaded(r), 1);
                mbar_init(bar_ready(r), 1);
                mbar_init(bar_rempty(r), W);
            }
            mbar_init(bar_comb, W);
            mbar_init_fence();
            mbar_arrive_expect_tx(bar_sched, a.smem_sched_bytes);
            for (uint32_t o = 0; o < a.smem_sched_bytes; o += 32768)
                bulk_g2s(smb + o, reinterpret_cast<const char *>(a.sched) + o, min(32768u, a.smem_sched_bytes - o),
                         bar_sched);
            if (!mbar_wait_bounded(bar_sched, 0, abort_flag, a.wait_ns)) {
                s_abort = 1;
                atomicOr(a.err, 1);
            }
        }
    }
    // the zero tile of each region (read by padding operations)
    for (uint32_t r = 0; r < a.n_buf; ++r)
        for (uint32_t i = threadIdx.x; i < PB / 16; i += blockDim.x)
            *reinterpret_cast<ulonglong2 *>(sm + lay.src0 + r * a.src_bytes + a.n_in * PB + i * 16) =
                make_ulonglong2(0, 0);
    __syncthreads();
    if (s_abort) return;
    mbar_try_wait(bar_sched, 0);  // completed: orders the copied schedule before this thread's reads

    // ------------------------------------------------------------------ stager
    if (warp == W) {
        const uint32_t bar_bytes = a.n_boxes * a.box_rows * TB;
        constexpr uint32_t kChunks = TB / 16;
        const uint32_t n_chunks = 2 * a.n_in * kChunks;
        uint32_t k = 0, armed = 0;  // tiles whose copies were issued
        for (uint32_t tile = blockIdx.x; tile < total; tile += gridDim.x, ++k) {
            const uint32_t r = a.n_buf == 2 ? (k & 1) : 0, ph = (a.n_buf == 2 ? k >> 1 : k) & 1;
            const uint32_t l = a.limb0 + tile / a.tiles_per_limb, k0 = (tile % a.tiles_per_limb) * T;
            const uint32_t dst = smb + lay.src0 + r * a.src_bytes;
            if (!mbar_wait_bounded(bar_rempty(r), ph ^ 1, abort_flag, a.wait_ns)) {
                fail();
                break;
            }
            if (lane == 0) {
                s_limb[r] = a.limbs[l];
                fence_proxy_async();
                const uint32_t extra = (a.flags & kWsFlagExtraTx) && k == 0 ? 16 : 0;
                mbar_arrive_expect_tx(bar_loaded(r), (a.n_in ? bar_bytes : 0) + extra);
                for (uint32_t j = 0; j < a.n_boxes; ++j) {
                    const uint32_t z = min(j * a.box_rows, 2 * a.n_in - a.box_rows);
                    tma_load_3d(dst + z * TB, &tm_in, k0, l, z, bar_loaded(r));
                }
            }
            armed = k + 1;
            if (SPLIT) {
                if (!mbar_wait_bounded(bar_loaded(r), ph, abort_flag, a.wait_ns)) {
                    fail();
                    break;
                }
                char *reg = sm + lay.src0 + r * a.src_bytes;
                uint32_t i = lane;
                for (; i + 96 < n_chunks; i += 128) {
                    ulonglong2 x[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) x[u] = *reinterpret_cast<const ulonglong2 *>(reg + (i + 32 * u) * 16);
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        *reinterpret_cast<ulonglong2 *>(reg + (i + 32 * u) * 16) =
                            make_ulonglong2(A::operand(x[u].x), A::operand(x[u].y));
                }
                for (; i < n_chunks; i += 32) {
                    ulonglong2 *q = reinterpret_cast<ulonglong2 *>(reg + i * 16);
                    const ulonglong2 x = *q;
                    *q = make_ulonglong2(A::operand(x.x), A::operand(x.y));
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_ready(r));
            }
        }
        // copies in flight land before the CTA exits
        if (lane == 0 && *abort_flag) {
            int never = 0;
            for (uint32_t j = 0; j < a.n_buf && j < armed; ++j) {
                const uint32_t kk = armed - 1 - j;
                const uint32_t r = a.n_buf == 2 ? (kk & 1) : 0, ph = (a.n_buf == 2 ? kk >> 1 : kk) & 1;
                mbar_wait_bounded(bar_loaded(r), ph, &never, kDrainNs);
            }
        }
        return;
    }

    // -------------------------------------------------------------- consumers
    const uint32_t lane_off = lane * VB;
    const uint32_t wt = a.o_warp + warp * kWarpTableWords;
    const uint32_t op0 = sw[wt] * 4, n_batches = sw[wt + 1] / P;
    const uint32_t seg0 = sw[wt + 2] * 4, tg0 = sw[wt + 3];
    const uint32_t ring_w = lay.ring0 + warp * D * P * TB + lane_off;  // byte offset in `sm`
    const uint32_t slots = lay.slot0 + sw[wt + 4] * PB + lane_off;  // this lane's words of its warp's slot 0
    const uint64_t pol = evict_first_policy();
    // the prefetch cursor: batch pf_b of tile pf_tile, D - 1 batches ahead;
    // pf_lb / pf_tb: the tile's limb of plaintext 0 and this lane's words in
    // it (byte pointers), recomputed when the cursor enters the next tile
    uint32_t pf_tile = blockIdx.x, pf_b = 0, pf_slot = 0;
    const char *pf_lb = nullptr, *pf_tb = nullptr;
    const uint64_t stride_bytes = (uint64_t)a.pt_stride * 8;
    auto pf_bases = [&]() {
        if (pf_tile >= total || !a.has_pt) return;
        const uint32_t l = a.limb0 + pf_tile / a.tiles_per_limb, k0 = (pf_tile % a.tiles_per_limb) * T;
        pf_lb = reinterpret_cast<const char *>(a.pt + (size_t)l * a.N);
        pf_tb = pf_lb + (k0 + lane * C) * 8;
    };
    pf_bases();
    auto prefetch = [&]() {
        if (n_batches && pf_tile < total && a.has_pt) {
            const uint4 ops = *reinterpret_cast<const uint4 *>(sm + op0 + pf_b * P * 4);
            const uint32_t o[4] = {ops.x, ops.y, ops.z, ops.w};
            const uint32_t dst = smb + ring_w + pf_slot * P * TB;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const bool cst = KC && (o[i] & kOpConst);
                const char *src = (cst ? pf_lb : pf_tb) + (uint64_t)(o[i] >> kOpPtShift) * stride_bytes;
                cp_async16(dst + i * TB, src, !(o[i] & kOpNop), pol);
            }
        }
        cp_async_commit();  // one group per batch, empty ones included
        if (++pf_slot == D) pf_slot = 0;
        if (n_batches && ++pf_b == n_batches) {
            pf_b = 0;
            pf_tile += gridDim.x;
            pf_bases();
        }
    };
#pragma unroll 1
    for (uint32_t i = 0; i + 1 < D; ++i) prefetch();

    uint32_t slot = 0, k = 0;
    for (uint32_t tile = blockIdx.x; tile < total; tile += gridDim.x, ++k) {
        const uint32_t r = a.n_buf == 2 ? (k & 1) : 0, ph = (a.n_buf == 2 ? k >> 1 : k) & 1;
        if (!mbar_wait_bounded(SPLIT ? bar_ready(r) : bar_loaded(r), ph, abort_flag, a.wait_ns)) {
            fail();
            cp_async_wait<0>();
            return;
        }
        const uint32_t l = a.limb0 + tile / a.tiles_per_limb;
        const uint32_t k0 = (tile % a.tiles_per_limb) * T;
        const uint32_t lim = smem_addr(&s_limb[r]);
        const uint32_t src = lay.src0 + r * a.src_bytes + lane_off;
        const uint32_t part_k = lay.part0 + (k & 1) * a.n_part * PB + lane_off;
        const uint64_t q = load_limb(lim).q;

        Acc acc[2][C];
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int x = 0; x < C; ++x) A::zero(acc[c][x]);
        uint32_t sp = seg0, tp = tg0;
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
                const uint32_t dst = part_k + (target & ~kPartBit) * PB;
                sts<C>(sm, dst, y0);
                sts<C>(sm, dst + TB, y1);
            } else {
                uint64_t *dst = a.out + ((size_t)target * 2 * a.L + l) * a.N + k0 + lane * C;
                stg<C>(dst, y0);
                stg<C>(dst + (size_t)a.L * a.N, y1);
            }
        };
        for (uint32_t b = 0; b < n_batches; ++b) {
            prefetch();                 // batch + D - 1 into the slot group freed last iteration
            cp_async_wait<D - 1>();     // this lane's copies of this batch have landed
            const uint4 h4 = *reinterpret_cast<const uint4 *>(sm + op0 + b * P * 4);
            const uint32_t hw[4] = {h4.x, h4.y, h4.z, h4.w};
            if (hw[0] & kOpFold) {
                const LimbConst m = load_limb(lim);
#pragma unroll
                for (int c = 0; c < 2; ++c)
#pragma unroll
                    for (int x = 0; x < C; ++x) A::fold(acc[c][x], m);
            }
            V<C> g0, g1;  // the signed sum of this batch's SEG (operand form)
            const bool seg = hw[0] & kOpSeg;
            if (seg) {
                // shared signed sums this warp forms for its own later uses
                // (Sec. 4.2 "Sharing Signed Sums"), then this group's sum
                const uint32_t nf = hw[0] & (kOpMaxSources - 1);
                for (uint32_t f = 0; f < nf; ++f) {
                    const uint32_t dst = slots + sw[sp >> 2] * PB;
                    V<C> u0, u1;
                    sp = signed_sum<SPLIT, C, TB>(sm, src, sp + 4, lim, slots, u0, u1);
                    if constexpr (SPLIT) {
#pragma unroll
                        for (int x = 0; x < C; ++x) {
                            u0.x[x] = A::operand(u0.x[x]);
                            u1.x[x] = A::operand(u1.x[x]);
                        }
                    }
                    sts<C>(sm, dst, u0);
                    sts<C>(sm, dst + TB, u1);
                }
                sp = signed_sum<SPLIT, C, TB>(sm, src, sp, lim, slots, g0, g1);
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    g0.x[x] = A::operand(g0.x[x]);
                    g1.x[x] = A::operand(g1.x[x]);
                }
            }
            const uint32_t rb = ring_w + slot * P * TB;
#pragma unroll
            for (uint32_t i = 0; i < P; ++i) {
                const uint32_t op = hw[i];
                V<C> pt = lds<C>(sm, rb + i * TB);
                if (KC && (op & kOpConst)) pt.x[1] = pt.x[0];  // a CONST plaintext: its limb's residue 0
                V<C> s0, s1;
                if (i == 0 && seg) {
                    s0 = g0;
                    s1 = g1;
                } else {
                    const uint32_t so = src + (op & (kOpMaxSources - 1)) * PB;
                    s0 = lds<C>(sm, so);
                    s1 = lds<C>(sm, so + TB);
                }
#pragma unroll
                for (int x = 0; x < C; ++x) {
                    const uint64_t gg = A::operand(pt.x[x]);
                    A::mac(acc[0][x], gg, s0.x[x]);
                    A::mac(acc[1][x], gg, s1.x[x]);
                }
            }
            if (++slot == D) slot = 0;
            if (hw[P - 1] & kOpLast) finish();
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar_rempty(r));  // this warp is done with region r

        // outputs split across warps: add the partial sums of this tile
        if (a.n_comb) {
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_comb);
            if (!mbar_wait_bounded(bar_comb, k & 1, abort_flag, a.wait_ns)) {
                fail();
                cp_async_wait<0>();
                return;
            }
            for (uint32_t rr = warp; rr < a.n_comb; rr += W) {
                V<C> y0{}, y1{};
                for (uint32_t pi = sw[a.o_comb_off + rr]; pi < sw[a.o_comb_off + rr + 1]; ++pi) {
                    const uint32_t ps = part_k + sw[a.o_comb_parts + pi] * PB;
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
    }
    cp_async_wait<0>();  // the prefetches past the last tile (empty groups) retire
}

template <bool NARROW, uint32_t MAXW>
void *select_ws_d(bool kc, uint32_t D)
{
    if (D == 3)
        return kc ? reinterpret_cast<void *>(&ws_kernel<NARROW, 4, true, MAXW, 3>)
                  : reinterpret_cast<void *>(&ws_kernel<NARROW, 4, false, MAXW, 3>);
    if (D == 4)
        return kc ? reinterpret_cast<void *>(&ws_kernel<NARROW, 4, true, MAXW, 4>)
                  : reinterpret_cast<void *>(&ws_kernel<NARROW, 4, false, MAXW, 4>);
    return nullptr;
}

// the variant for W consumer warps and a ring of D groups: up to fifteen
// consumer warps and the stager have 128 registers a thread, sixteen 96
void *select_ws(bool narrow, uint32_t P, bool kc, uint32_t W, uint32_t D)
{
    if (P != 4 || W == 0 || W > kWsMaxWarps) return nullptr;
    if (W > 15) return narrow ? select_ws_d<true, 16>(kc, D) : select_ws_d<false, 16>(kc, D);
    return narrow ? select_ws_d<true, 15>(kc, D) : select_ws_d<false, 15>(kc, D);
}

}  // namespace

int ws_kernel_attributes(bool narrow, uint32_t P, bool kc, uint32_t W, uint32_t D, cudaFuncAttributes *attr)
{
    void *fn = select_ws(narrow, P, kc, W, D);
    if (!fn) return set_error(FIONA_ERR_ARG, "warp-specialised kernel: no variant with P=%u", P);
    cudaError_t e = cudaFuncGetAttributes(attr, fn);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "ws kernel attributes: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

int ws_configure_kernel(bool narrow, uint32_t P, bool kc, uint32_t W, uint32_t D, size_t smem)
{
    void *fn = select_ws(narrow, P, kc, W, D);
    if (!fn) return set_error(FIONA_ERR_ARG, "warp-specialised kernel: no variant with P=%u", P);
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "ws kernel attribute: %s", cudaGetErrorString(e));
    return FIONA_OK;
}

// kernel_tiled.cu
int input_tensor_map(uint32_t N, uint32_t layout_L, uint32_t n_in, uint32_t T, uint32_t box_rows,
                     const uint64_t *in, CUtensorMap *tm);

int launch_ws(const fiona_plan *p, void *stream, const uint64_t *in, const uint64_t *pt, uint64_t *out, uint32_t l0,
              uint32_t l1, uint32_t layout_L)
{
    const TiledSchedule *ts = p->tiled;
    if (l1 <= l0) return FIONA_OK;
    WsArgs a = ts->ws_args;
    a.in = in;
    a.pt = pt;
    a.out = out;
    a.limb0 = l0;
    a.n_limbs = l1 - l0;
    a.L = layout_L;
    a.pt_stride = layout_L * a.N;
    const uint32_t tiles = a.n_limbs * a.tiles_per_limb;
    const uint32_t resident = ts->ctas_per_sm * (uint32_t)std::max(p->ctx->sm_count, 1);
    dim3 grid(std::min(tiles, resident));
    dim3 block((ts->warps + 1) * 32);
    void *fn = select_ws(ts->narrow, ts->batch, ts->has_const, ts->warps, ts->ring);
    if (!fn) return set_error(FIONA_ERR_INTERNAL, "ws kernel: no variant for the schedule's shape");
    CUtensorMap tm;
    if (const int rc = input_tensor_map(a.N, layout_L, a.n_in, T, a.box_rows, in, &tm)) return rc;
    void *args[] = {&a, &tm};
    cudaError_t e = cudaLaunchKernel(fn, grid, block, args, ts->smem, (cudaStream_t)stream);
    if (e != cudaSuccess) return set_error(FIONA_ERR_CUDA, "ws kernel launch: %s", cudaGetErrorString(e));
    return FIONA_OK;
}
