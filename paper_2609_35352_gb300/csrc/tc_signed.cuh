// tc_signed.cuh -- the signed sums of a tile as one contraction on the 5th
// generation tensor cores (tcgen05), for layers whose moduli are all below
// 2^50 and that run one coefficient per lane (T = 32).
//
// All scale groups' signed sums of a tile (Sec. 4.2 "Grouping
// Reconstruction Operations") form the product S = A W of the tile's inputs
// A (rows: the 64 (poly, coefficient) pairs; columns: the inputs) and the
// layer's weight matrix W (inputs x groups: each input's net sign in the
// group, t in {-1, 0, +1}, or a small integer where expanded shared sums
// repeat an input).  Residues have 50 bits; each is cut into five 10-bit
// chunks v, held exactly in fp16 as 1024 + v (exponent of 1024, mantissa
// v), so
//   S = sum_j 2^(10 j) (A_j W - 1024 * colsum(W))
// where A_j holds chunk j.  The tensor cores compute each A_j W with f32
// accumulation, exact because every partial sum is an integer below 2^24
// (at most 2047 * sum |w| over a group; the lowering checks the bound).  The
// chunk matrices go to tensor memory
// (TMEM, the A operand; M = 64 rows, 16 rows per warp quarter: row 16 q + l
// in lane 32 q + l), W sits in shared memory in the canonical K-major layout
// without swizzle (core matrices of 8 rows x 16 bytes), and each D_j = A_j W
// (64 x N, f32) lands in TMEM.
//
// The column layout and W's layout are in tc_geometry.h.
#pragma once
#include <stdint.h>

#include "tc_geometry.h"
#include "tile_math.cuh"

namespace tcs {

constexpr uint32_t kChunks = kTcChunks;
constexpr uint32_t kFp16Bias = 0x6400;  // fp16 bits of 1024.0

// `cols` columns of tensor memory (a power of two, 32 to 512) for the CTA,
// their address written to shared memory at `dst_smem`; one warp allocates
// and later frees them.
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t cols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t cols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(cols) : "memory");
}

__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// four 32-bit columns of this warp's lanes from the TMEM address `taddr`
// (lane << 16 | column)
__device__ __forceinline__ void st4(uint32_t taddr, const uint32_t (&v)[4])
{
    asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1, %2, %3, %4};" ::"r"(taddr), "r"(v[0]), "r"(v[1]),
                 "r"(v[2]), "r"(v[3])
                 : "memory");
}

__device__ __forceinline__ void wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// four 32-bit columns of this warp's lanes from `taddr` (complete after wait_ld)
__device__ __forceinline__ void ld4(uint32_t taddr, uint32_t (&v)[4])
{
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3])
                 : "r"(taddr)
                 : "memory");
}

__device__ __forceinline__ void wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Shared-memory descriptor of a K-major operand without swizzle: start
// address, LBO = byte stride between core matrices along K, SBO = byte
// stride between groups of 8 rows; version 1 (bits 46-47).
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    return (uint64_t)((addr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46);
}

// Instruction descriptor, kind::f16: D f32, A and B f16, both K-major.
__host__ __device__ constexpr uint32_t idesc_f16(uint32_t M, uint32_t N)
{
    return (1u << 4) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

// D (TMEM) = or += A (TMEM) x B (shared memory, descriptor), M = 64, K = 16
__device__ __forceinline__ void mma(uint32_t d, uint32_t a, uint64_t bdesc, uint32_t idesc, uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
        "r"(a), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// the mbarrier at `bar` gets one arrival when this thread's earlier MMAs complete
__device__ __forceinline__ void commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// Chunk j of two residues a, b (below 2^50) as a pair of fp16 values
// 1024 + chunk, a in the low half.
template <int J>
__device__ __forceinline__ uint32_t chunk_pair(uint64_t a, uint64_t b)
{
    const uint32_t alo = (uint32_t)a, ahi = (uint32_t)(a >> 32), blo = (uint32_t)b, bhi = (uint32_t)(b >> 32);
    uint32_t g;
    if constexpr (J == 0) {
        g = __byte_perm(alo, blo, 0x5410);  // bits 0-15 of each
    } else if constexpr (J == 1) {
        g = __byte_perm(alo, blo, 0x6521) >> 2;  // bits 8-23 of each, then 10-19 at the bottom of each half
    } else if constexpr (J == 2) {
        g = __byte_perm(alo, blo, 0x7632) >> 4;  // bits 16-31, then 20-29
    } else if constexpr (J == 3) {
        const uint32_t x = __funnelshift_r(alo, ahi, 30), y = __funnelshift_r(blo, bhi, 30);  // bits 30-61
        g = __byte_perm(x, y, 0x5410);
    } else {
        g = __byte_perm(ahi, bhi, 0x6521);  // bits 40-55 of each: 40-49 at the bottom of each half
    }
    return (g & 0x03FF03FFu) | (kFp16Bias | (kFp16Bias << 16));
}

// Chunk j of the 8 residues x as four fp16 pairs, stored to the 4 TMEM
// columns at `taddr` (this warp's lanes).
template <int J>
__device__ __forceinline__ void store_chunk(uint32_t taddr, const uint64_t (&x)[8])
{
    uint32_t v[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) v[m] = chunk_pair<J>(x[2 * m], x[2 * m + 1]);
    st4(taddr, v);
}

// The tile row of TMEM lane l of quarter q with M = 64: poly q / 2,
// coefficient 16 (q % 2) + l, for l < 16 (lanes 16-31 of a quarter are not
// read by the contraction).
__device__ __forceinline__ uint32_t row_poly(uint32_t q) { return q >> 1; }
__device__ __forceinline__ uint32_t row_coef(uint32_t q, uint32_t lane) { return 16 * (q & 1) + (lane & 15); }

// This warp's share of the chunk matrices: the warp reads TMEM quarter q
// (its warp index mod 4) and takes every nq-th group of 8 inputs from the
// kq-th.  `src` = byte offset in `sm` of this lane's word of input 0 (its
// row's poly and coefficient), `pb` = bytes between inputs; inputs from
// n_in on are zero.
__device__ __forceinline__ void convert(const char *sm, uint32_t src, uint32_t pb, uint32_t n_in, const TcGeometry &g,
                                        uint32_t tmem_q, uint32_t kq, uint32_t nq)
{
    for (uint32_t b = kq; b < g.K / 8; b += nq) {
        uint64_t x[8];
#pragma unroll
        for (uint32_t i = 0; i < 8; ++i) {
            const uint32_t k = 8 * b + i;
            x[i] = k < n_in ? *reinterpret_cast<const uint64_t *>(sm + src + k * pb) : 0;
        }
        const uint32_t t = tmem_q + 4 * b;
        store_chunk<0>(t + g.a_col(0), x);
        store_chunk<1>(t + g.a_col(1), x);
        store_chunk<2>(t + g.a_col(2), x);
        store_chunk<3>(t + g.a_col(3), x);
        store_chunk<4>(t + g.a_col(4), x);
    }
}

// The contraction, issued by one thread: D_j = A_j W for every chunk, K in
// steps of 16; completion arrives on the mbarrier `bar`.  `w_addr` = shared
// address of W (16-byte aligned).
__device__ __forceinline__ void issue(uint32_t tmem, uint32_t w_addr, const TcGeometry &g, uint32_t bar)
{
    const uint32_t id = idesc_f16(64, g.N);
#pragma unroll 1
    for (uint32_t j = 0; j < kChunks; ++j)
#pragma unroll 1
        for (uint32_t s = 0; s < g.K / 16; ++s)
            mma(tmem + g.d_col(j), tmem + g.a_col(j) + 8 * s, smem_desc(w_addr + 256 * s, 128, g.sbo()), id, s > 0);
    commit(bar);
}

// fp32 bits of 1.5 * 2^23 + e for an integer |e| < 2^22
constexpr uint32_t kMagicBits = 0x4B400000u;
// sum over the chunks of kMagicBits * 2^(10 j), mod 2^64
constexpr uint64_t kMagicSum =
    (uint64_t)kMagicBits * (1ull + (1ull << 10) + (1ull << 20) + (1ull << 30) + (1ull << 40));

// S mod q from the five chunk products of one (row, group): d_j = A_j W at
// the row and group, `magic` = 1.5 * 2^23 - 1024 * (sum of the group's
// weights), `bias` = a multiple of q above |S|.  Each d_j + magic is exact
// (an integer below 2^24), its bits minus kMagicBits are the chunk's signed
// sum e_j, and S = sum_j 2^(10 j) e_j; the sum is formed mod 2^64, where
// S + bias is its true value.
__device__ __forceinline__ uint64_t combine(const uint32_t (&d)[kChunks], float magic, uint64_t bias,
                                            const LimbConst &m)
{
    uint64_t u = bias - kMagicSum;
#pragma unroll
    for (uint32_t j = 0; j < kChunks; ++j)
        u += (uint64_t)__float_as_uint(__fadd_rn(__uint_as_float(d[j]), magic)) << (10 * j);
    return rns::reduce64(u, m);
}

// This warp's share of the epilogue: every nq-th run of 4 groups from the
// kq-th, read from its TMEM quarter; each lane below 16 passes its row's
// residues S mod q to put(group, value).  `magic` = the groups' constants
// (shared memory).
template <class Put>
__device__ __forceinline__ void epilogue(uint32_t tmem_q, const TcGeometry &g, uint32_t n_groups, const float *magic,
                                         uint64_t bias, const LimbConst &m, uint32_t lane, uint32_t kq, uint32_t nq,
                                         Put put)
{
    for (uint32_t g4 = 4 * kq; g4 < n_groups; g4 += 4 * nq) {
        uint32_t d[kChunks][4];
#pragma unroll
        for (uint32_t j = 0; j < kChunks; ++j) ld4(tmem_q + g.d_col(j) + g4, d[j]);
        wait_ld();
#pragma unroll
        for (uint32_t i = 0; i < 4; ++i) {
            const uint32_t gi = g4 + i;
            if (gi < n_groups && lane < 16) {
                const uint32_t e[kChunks] = {d[0][i], d[1][i], d[2][i], d[3][i], d[4][i]};
                put(gi, combine(e, magic[gi], bias, m));
            }
        }
    }
}

}  // namespace tcs
